// Causal self-attention with grouped KV heads over the compacted sequence or
// the text-only KV cache (DecoMoE Section 3.2: once the visual block exits,
// attention in that layer and every later one runs on the shortened text-only
// sequence; Algorithm 2, last step: decoding reuses the shortened cache;
// Appendix FLOPs 2qS(S+1) per prefill layer and 4qC per decode forward).
//
// Layouts: q [n, Hq, D], k and v [C, Hkv, D] (one layer slice of the KV
// caches the visual-block removal compacts), out [n, Hq, D], all bf16,
// D = 128. Query i is at position C - n + i and sees keys 0 .. C - n + i;
// query head h reads KV head h / (Hq / Hkv).
//
// Decode sizes (few queries per KV head): split-key partials. CTA (s, g)
// takes one chunk of keys (32 to 128) of KV head g and every query of its
// head group: K and V chunk rows staged in shared memory (cp.async), one warp
// per query, scores and weighted values on CUDA cores with fp32 accumulation;
// the chunk's softmax maximum, sum and weighted value row go out as partials
// and a second launch combines the partials of each query in a fixed order
// (deterministic).
#include <cfloat>

#include "decomoe_internal.cuh"

namespace decomoe {

constexpr int ATT_D = 128;
constexpr int ATT_CH_MAX = 128;                 // keys per split (at most)
constexpr int ATT_THREADS = 256;                // 8 warps: one query at a time each
constexpr int ATT_KROW = ATT_D * 2 + 16;        // padded K row in shared memory (bytes): conflict-free 16-byte reads
constexpr int ATT_MAXQ = 64;                    // queries per KV head handled by one split CTA
constexpr int ATT_PROW = ATT_D + 4;             // floats per partial row: acc[D], m, l, 2 unused (16-byte rows)

struct AttArgs {
  const uint4* q;   // [n, Hq, D]
  const uint4* k;   // [C, Hkv, D]
  const uint4* v;
  int64_t n, C;
  int Hq, Hkv, nsplit, chunk;
  float scale;
  float* part;      // [nsplit][Hkv][nq][ATT_PROW]: acc[D], m, l
};

__host__ __device__ constexpr size_t att_split_smem() {
  return static_cast<size_t>(ATT_CH_MAX) * ATT_KROW + static_cast<size_t>(ATT_CH_MAX) * ATT_D * 2 +
         static_cast<size_t>(ATT_MAXQ) * ATT_D * 2;
}

// Keys per split: 128 when that already gives a CTA per SM, else smaller
// chunks (multiples of 32) so that short caches still spread over the SMs.
static int att_chunk(int64_t C, int Hkv) {
  const int64_t want = std::max<int64_t>(1, sm_count() / std::max(1, Hkv));
  int64_t ch = (C + want - 1) / want;
  ch = (ch + 31) / 32 * 32;
  return static_cast<int>(std::min<int64_t>(ATT_CH_MAX, std::max<int64_t>(32, ch)));
}

// nq = n * (Hq / Hkv) <= ATT_MAXQ queries of KV head g against one key chunk
// (query qi = i * G + j is head g * G + j of token i). Warp w takes queries
// w, w + 8, ...: lane l owns keys l, l + 32, ... for the scores (the query's
// 32-feature slices held in registers, the key rows read from shared
// memory), then features 4l .. 4l + 3 for the weighted value rows (each key's
// weight passed from its lane by a shuffle).
__global__ void __launch_bounds__(ATT_THREADS)
    k_attn_split(const AttArgs a) {
  pdl_enter();
  extern __shared__ uint8_t smem[];
  const int s = blockIdx.x, g = blockIdx.y;
  const int G = a.Hq / a.Hkv;
  const int nq = static_cast<int>(a.n) * G;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint8_t* sK = smem;                                                          // [CH][KROW]
  const __nv_bfloat16* sV = reinterpret_cast<const __nv_bfloat16*>(sK + ATT_CH_MAX * ATT_KROW);  // [CH][D]
  uint4* sQ = reinterpret_cast<uint4*>(sK + ATT_CH_MAX * ATT_KROW + ATT_CH_MAX * ATT_D * 2);     // [nq][D] bf16
  const int64_t c0 = static_cast<int64_t>(s) * a.chunk;
  const int nk = static_cast<int>(a.C - c0 < a.chunk ? a.C - c0 : a.chunk);
  constexpr int VPR = ATT_D / 8;  // 16-byte vectors per head row
  // stage this chunk's K and V rows of head g (16-byte copies, all in flight)
  for (int i = tid; i < nk * VPR; i += ATT_THREADS) {
    const int r = i / VPR, c = i - r * VPR;
    const int64_t src = ((c0 + r) * a.Hkv + g) * VPR + c;
    cp_async16(smem_u32(sK + r * ATT_KROW + c * 16), a.k + src);
    cp_async16(smem_u32(const_cast<__nv_bfloat16*>(sV) + r * ATT_D + c * 8), a.v + src);
  }
  // and the group's query rows (query qi = i * G + j is head g * G + j of token i)
  for (int i = tid; i < nq * VPR; i += ATT_THREADS) {
    const int qi = i / VPR, c = i - qi * VPR;
    const int ti = qi / G, hj = qi - ti * G;
    cp_async16(smem_u32(sQ + i), a.q + (static_cast<int64_t>(ti) * a.Hq + g * G + hj) * VPR + c);
  }
  cp_async_wait_all();
  __syncthreads();
  float* part = a.part + (static_cast<int64_t>(s) * a.Hkv + g) * nq * ATT_PROW;
  for (int qi = warp; qi < nq; qi += ATT_THREADS / 32) {
    const int ti = qi / G;
    const uint4* qrow = sQ + qi * VPR;
    const int64_t last = a.C - a.n + ti;  // the query's position: keys up to it are visible
    // scores of keys lane, lane + 32, lane + 64, lane + 96
    float sc[ATT_CH_MAX / 32];
#pragma unroll
    for (int u = 0; u < ATT_CH_MAX / 32; ++u) sc[u] = 0.f;
#pragma unroll
    for (int c4 = 0; c4 < VPR; c4 += 4) {
      // 32 features of the query (four 16-byte vectors, the same for every lane)
      float qf[32];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const uint4 u = qrow[c4 + c];
        qf[8 * c + 0] = bf16_lo(u.x); qf[8 * c + 1] = bf16_hi(u.x);
        qf[8 * c + 2] = bf16_lo(u.y); qf[8 * c + 3] = bf16_hi(u.y);
        qf[8 * c + 4] = bf16_lo(u.z); qf[8 * c + 5] = bf16_hi(u.z);
        qf[8 * c + 6] = bf16_lo(u.w); qf[8 * c + 7] = bf16_hi(u.w);
      }
#pragma unroll
      for (int u = 0; u < ATT_CH_MAX / 32; ++u) {
        const int t = lane + 32 * u;
        if (t < nk) {
          const uint4* kr = reinterpret_cast<const uint4*>(sK + t * ATT_KROW) + c4;
          float acc = sc[u];
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const uint4 kv = kr[c];
            acc = fmaf(bf16_lo(kv.x), qf[8 * c + 0], acc);
            acc = fmaf(bf16_hi(kv.x), qf[8 * c + 1], acc);
            acc = fmaf(bf16_lo(kv.y), qf[8 * c + 2], acc);
            acc = fmaf(bf16_hi(kv.y), qf[8 * c + 3], acc);
            acc = fmaf(bf16_lo(kv.z), qf[8 * c + 4], acc);
            acc = fmaf(bf16_hi(kv.z), qf[8 * c + 5], acc);
            acc = fmaf(bf16_lo(kv.w), qf[8 * c + 6], acc);
            acc = fmaf(bf16_hi(kv.w), qf[8 * c + 7], acc);
          }
          sc[u] = acc;
        }
      }
    }
    // softmax partials over the chunk's visible keys
    float mx = -FLT_MAX;
#pragma unroll
    for (int u = 0; u < ATT_CH_MAX / 32; ++u) {
      const int t = lane + 32 * u;
      const bool vis = t < nk && c0 + t <= last;
      sc[u] = vis ? sc[u] * a.scale : -FLT_MAX;
      mx = fmaxf(mx, sc[u]);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    float sum = 0.f;
#pragma unroll
    for (int u = 0; u < ATT_CH_MAX / 32; ++u) {
      sc[u] = sc[u] == -FLT_MAX ? 0.f : __expf(sc[u] - mx);
      sum += sc[u];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
    // weighted value rows: lane l sums features 4l .. 4l + 3 over the keys
    float o[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int u = 0; u < ATT_CH_MAX / 32; ++u) {
      const int tb = 32 * u;
      const int nt = nk - tb < 32 ? nk - tb : 32;
      for (int j = 0; j < nt; ++j) {
        const float p = __shfl_sync(0xffffffffu, sc[u], j);
        const uint2 vv = *reinterpret_cast<const uint2*>(sV + (tb + j) * ATT_D + 4 * lane);
        o[0] = fmaf(p, bf16_lo(vv.x), o[0]);
        o[1] = fmaf(p, bf16_hi(vv.x), o[1]);
        o[2] = fmaf(p, bf16_lo(vv.y), o[2]);
        o[3] = fmaf(p, bf16_hi(vv.y), o[3]);
      }
    }
    float* pr = part + qi * ATT_PROW;
    *reinterpret_cast<float4*>(pr + 4 * lane) = make_float4(o[0], o[1], o[2], o[3]);
    if (lane == 0) {
      pr[ATT_D] = sum > 0.f ? mx : -FLT_MAX;
      pr[ATT_D + 1] = sum;
    }
  }
  pdl_trigger();
}

// out[i, h, :] = sum_s e^(m_s - M) acc_s / sum_s e^(m_s - M) l_s over the
// splits s (M = max m_s). Block (token i x head h, 32-feature slice), 32
// warps: warp w sums the splits s = w, w + 32, ... in order (lane = feature),
// then the warp sums are added in warp order: a fixed order, so the result
// does not depend on timing, and each pass is about one round of loads.
constexpr int ATT_MAX_SPLITS = 1024;
constexpr int ATT_CWARPS = 32;
__global__ void __launch_bounds__(32 * ATT_CWARPS)
    k_attn_combine(const float* __restrict__ part, int64_t n, int Hq, int Hkv, int nsplit,
                   __nv_bfloat16* __restrict__ out) {
  pdl_enter();
  __shared__ float s_m[ATT_CWARPS], s_num[ATT_CWARPS][32], s_den[ATT_CWARPS];
  const int64_t ih = blockIdx.x;  // token i * Hq + head h
  const int64_t i = ih / Hq;
  const int h = static_cast<int>(ih - i * Hq);
  const int G = Hq / Hkv;
  const int g = h / G;
  const int nq = static_cast<int>(n) * G;
  const int qi = static_cast<int>(i) * G + (h - g * G);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int d = blockIdx.y * 32 + lane;
  auto prow = [&](int s) { return part + ((static_cast<int64_t>(s) * Hkv + g) * nq + qi) * ATT_PROW; };
  float mx = -FLT_MAX;
  for (int s = warp; s < nsplit; s += ATT_CWARPS) mx = fmaxf(mx, __ldg(prow(s) + ATT_D));
  if (lane == 0) s_m[warp] = mx;
  __syncthreads();
  float M = s_m[0];
#pragma unroll
  for (int w = 1; w < ATT_CWARPS; ++w) M = fmaxf(M, s_m[w]);
  float num = 0.f, den = 0.f;
  for (int s = warp; s < nsplit; s += ATT_CWARPS) {
    const float* p = prow(s);
    const float ms = __ldg(p + ATT_D);
    const float ls = __ldg(p + ATT_D + 1);
    const float as = __ldg(p + d);
    const float w = ms == -FLT_MAX ? 0.f : __expf(ms - M);  // no visible key in this split: weight 0
    num = fmaf(w, as, num);
    den = fmaf(w, ls, den);
  }
  s_num[warp][lane] = num;
  if (lane == 0) s_den[warp] = den;
  __syncthreads();
  if (warp == 0) {
    float a = s_num[0][lane], b = s_den[0];
#pragma unroll
    for (int w = 1; w < ATT_CWARPS; ++w) {
      a += s_num[w][lane];
      b += s_den[w];
    }
    out[ih * ATT_D + d] = __float2bfloat16_rn(a / b);
  }
}

// ------------------------------------------------------------------ prefill (tensor cores)
// Many queries per KV head (the compacted sequence's prefill): flash-style
// attention on tcgen05. A CTA takes one tile of 128 query rows for two query
// heads of the same KV group, so each K and V block it streams serves both.
// Per block j of 64 keys and head x: S_x = Q_x K_j^T (M = 128 queries, N = 64
// keys, K = 128 features) into tensor memory; four warps per head (one query
// row per thread) take the row maximum, write p = 2^(s*scale*log2e - m) as
// bf16 into tensor memory (the A operand of the next product) and add p to
// the row sum l; then O_x += P_x V_j (N = 128 features, K = 64 keys, V
// transposed beforehand so that the B operand is K-major) accumulates in
// tensor memory. The reference maximum m of a row moves only when the block
// maximum exceeds it by more than 8 (a factor 256): then that row's O and l
// are scaled by 2^(m_old - m_new) before the next product (otherwise p stays
// below 256, well inside bf16 and fp32); the final output is O / l either
// way. Tensor-core work of one head overlaps the other head's softmax: the
// issue order is PV_0(j), S_0(j+1), PV_1(j), S_1(j+1). Warp 0 streams K_j and
// V_j^T blocks by TMA into a four-stage ring; warp 1 issues the MMAs. Every
// wait is bounded; on a timeout the CTA records DECOMOE_ERR_TIMEOUT, lets its
// copies and MMAs land, frees its tensor memory and returns.
constexpr int ATP_BM = 128;                 // query rows per CTA
constexpr int ATP_BN = 64;                  // keys per block
constexpr int ATP_HEADS = 2;                // query heads per CTA (same KV head)
constexpr int ATP_NST = 4;                  // K / V ring stages
constexpr int ATP_QHALF = 128 * 64 * 2;     // Q: 128 rows x 64 features, 128-byte swizzle (16 KB)
constexpr int ATP_KHALF = ATP_BN * 64 * 2;  // K block: 64 keys x 64 features (8 KB)
constexpr int ATP_VT = 128 * ATP_BN * 2;    // V^T block: 128 features x 64 keys (16 KB)
constexpr int ATP_STAGE = 2 * ATP_KHALF + ATP_VT;
constexpr int ATP_THREADS = 64 + ATP_HEADS * 128;
constexpr int ATP_TMEM_COLS = 512;          // per head: S [0,64), P [64,96), O [128,256)
constexpr float ATP_RESCALE = 8.0f;         // log2 of the largest unnormalised p
constexpr size_t ATP_SMEM = 1024 + ATP_HEADS * 2 * ATP_QHALF + ATP_NST * ATP_STAGE + 32 * 8 + 16;

struct AttPreArgs {
  int64_t n, C;        // queries (the last n positions), keys
  int Hq, group;       // query heads, query heads per KV head
  float scale_log2;    // scale * log2(e)
  __nv_bfloat16* out;  // [n, Hq, D]
  int32_t* status;
  uint64_t limit_ns;
};

// vt[g][d][s] = v[s][g][d] for s < C, 0 up to C_pad (pad columns must be
// finite: their weights are zero)
__global__ void __launch_bounds__(256)
    k_attn_vt(const __nv_bfloat16* __restrict__ v, int64_t C, int Hkv, int64_t C_pad, __nv_bfloat16* __restrict__ vt) {
  pdl_enter();
  __shared__ __nv_bfloat16 tile[32][33];
  const int64_t s0 = static_cast<int64_t>(blockIdx.x) * 32;
  const int d0 = blockIdx.y * 32, g = blockIdx.z;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8
  for (int r = ty; r < 32; r += 8) {
    const int64_t s = s0 + r;
    tile[r][tx] = s < C ? v[(s * Hkv + g) * ATT_D + d0 + tx] : __float2bfloat16_rn(0.f);
  }
  __syncthreads();
  for (int r = ty; r < 32; r += 8) {
    const int64_t s = s0 + tx;
    if (s < C_pad) vt[(static_cast<int64_t>(g) * ATT_D + d0 + r) * C_pad + s] = tile[tx][r];
  }
}

// D(tmem) (+)= A(tmem) * B(smem desc)^T: A is 128 rows (lanes) x 16 bf16
// (8 columns, two elements per 32-bit column, the lower index in the low half).
__device__ __forceinline__ void tc_mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// Values loaded by tcgen05.ld are defined only after tcgen05.wait::ld: route
// them through an empty asm placed after the wait so no use moves above it.
template <int N>
__device__ __forceinline__ void after_wait(uint32_t (&r)[N]) {
#pragma unroll
  for (int i = 0; i < N; ++i) asm volatile("" : "+r"(r[i]));
}
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(ATP_THREADS, 1)
    k_attn_prefill(const __grid_constant__ CUtensorMap tma_q, const __grid_constant__ CUtensorMap tma_k,
                   const __grid_constant__ CUtensorMap tma_vt, const AttPreArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sQ = raw + pad;                              // [head][feature half]
  const uint32_t sKV = sQ + ATP_HEADS * 2 * ATP_QHALF;        // [stage]{K half 0, K half 1, V^T}
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + ATP_HEADS * 2 * ATP_QHALF + ATP_NST * ATP_STAGE);
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(bars + 32);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  const uint32_t bar0 = smem_u32(bars);
  const uint32_t Q_BAR = bar0, DRAIN = bar0 + 8;
  auto S_FULL = [&](int x) { return bar0 + 16u + 8u * x; };
  auto P_FULL = [&](int x) { return bar0 + 32u + 8u * x; };
  auto O_FINAL = [&](int x) { return bar0 + 48u + 8u * x; };
  auto FULL = [&](int st) { return bar0 + 64u + 8u * st; };
  auto EMPTY = [&](int st) { return bar0 + 96u + 8u * st; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int npair = a.Hq / ATP_HEADS;
  const int ntile = static_cast<int>((a.n + ATP_BM - 1) / ATP_BM);
  // heaviest tiles (most key blocks) first
  const int hp = blockIdx.x % npair;
  const int qt = ntile - 1 - static_cast<int>(blockIdx.x / npair);
  const int h0 = hp * ATP_HEADS;
  const int g = h0 / a.group;  // both heads read KV head g (the group size is even)
  const int64_t p0 = a.C - a.n + static_cast<int64_t>(qt) * ATP_BM;  // position of the tile's first row
  const int64_t last = p0 + ATP_BM - 1 < a.C - 1 ? p0 + ATP_BM - 1 : a.C - 1;
  const int nblk = static_cast<int>(last / ATP_BN) + 1;  // key blocks any row of the tile can see

  if (threadIdx.x == 0) {
    *s_abort = 0;
    mbar_init(Q_BAR, 1);
    mbar_init(DRAIN, 1);
    for (int x = 0; x < ATP_HEADS; ++x) {
      mbar_init(S_FULL(x), 1);
      mbar_init(P_FULL(x), 128);
      mbar_init(O_FINAL(x), 1);
    }
    for (int st = 0; st < ATP_NST; ++st) {
      mbar_init(FULL(st), 1);
      mbar_init(EMPTY(st), 1);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<uint32_t*>(s_tmem)), ATP_TMEM_COLS);
    tmem_relinquish();
  }
  pdl_wait();  // q, k and the transposed v are ready
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  auto S_TM = [&](int x) { return tmem + 256u * x; };
  auto P_TM = [&](int x) { return tmem + 256u * x + 64u; };
  auto O_TM = [&](int x) { return tmem + 256u * x + 128u; };
  constexpr uint32_t IDESC_S = idesc_bf16_f32(ATP_BM, ATP_BN);
  constexpr uint32_t IDESC_O = idesc_bf16_f32(ATP_BM, ATT_D);

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0)
    if (lane == 0) {
      tma_prefetch_desc(&tma_q);
      tma_prefetch_desc(&tma_k);
      tma_prefetch_desc(&tma_vt);
      bool ok = true;
      uint32_t armed = 0, armed_ph = 0;
      mbar_arrive_expect_tx(Q_BAR, ATP_HEADS * 2 * ATP_QHALF);
      const int qrow0 = qt * ATP_BM;
      for (int x = 0; x < ATP_HEADS; ++x)
        for (int kb = 0; kb < 2; ++kb) tma_load_3d(sQ + (2 * x + kb) * ATP_QHALF, &tma_q, Q_BAR, 64 * kb, h0 + x, qrow0);
      for (int j = 0; j < nblk; ++j) {
        const int st = j % ATP_NST;
        const uint32_t ph = (j / ATP_NST) & 1;
        if (!mbar_wait(EMPTY(st), ph ^ 1u, a.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(FULL(st), ATP_STAGE);
        const int key0 = j * ATP_BN;
        const uint32_t base = sKV + st * ATP_STAGE;
        tma_load_3d(base, &tma_k, FULL(st), 0, g, key0);
        tma_load_3d(base + ATP_KHALF, &tma_k, FULL(st), 64, g, key0);
        tma_load_3d(base + 2 * ATP_KHALF, &tma_vt, FULL(st), key0, 0, g);
        armed |= 1u << st;
        armed_ph = (armed_ph & ~(1u << st)) | (ph << st);
      }
      if (!ok) {
        *s_abort = 1;
        report_status(a.status, DECOMOE_ERR_TIMEOUT);
        int no_abort = 0;
        mbar_wait(Q_BAR, 0, a.limit_ns, &no_abort);
        for (int st = 0; st < ATP_NST; ++st)
          if ((armed >> st) & 1u) mbar_wait(FULL(st), (armed_ph >> st) & 1u, a.limit_ns, &no_abort);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (lane 0)
    if (lane == 0) {
      // S_x = Q_x K^T over the 128 features (two 64-feature halves)
      auto issue_s = [&](int x, int st) {
        const uint32_t base = sKV + st * ATP_STAGE;
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint64_t ad = smem_desc_kmajor<64>(sQ + (2 * x + kb) * ATP_QHALF);
          const uint64_t bd = smem_desc_kmajor<64>(base + kb * ATP_KHALF);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_f16(S_TM(x), ad + 2u * kk, bd + 2u * kk, IDESC_S, (kb | kk) != 0 ? 1u : 0u);
        }
      };
      // O_x += P_x V_j over the block's 64 keys
      auto issue_pv = [&](int x, int st, bool acc) {
        const uint64_t bd = smem_desc_kmajor<64>(sKV + st * ATP_STAGE + 2 * ATP_KHALF);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_f16_ts(O_TM(x), P_TM(x) + 8u * kk, bd + 2u * kk, IDESC_O, (acc || kk > 0) ? 1u : 0u);
      };
      bool ok = mbar_wait(Q_BAR, 0, a.limit_ns, s_abort) && mbar_wait(FULL(0), 0, a.limit_ns, s_abort);
      bool issued = false;
      if (ok) {
        tc_fence_after();
        for (int x = 0; x < ATP_HEADS; ++x) {
          issue_s(x, 0);
          tc_commit(S_FULL(x));
        }
        issued = true;
      }
      for (int j = 0; ok && j < nblk; ++j) {
        const int st = j % ATP_NST;
        for (int x = 0; x < ATP_HEADS; ++x) {
          if (!mbar_wait(P_FULL(x), j & 1, a.limit_ns, s_abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_pv(x, st, j > 0);
          if (x == ATP_HEADS - 1) tc_commit(EMPTY(st));  // K_j and V_j read by every product
          if (j + 1 < nblk) {
            const int st1 = (j + 1) % ATP_NST;
            if (x == 0) {
              if (!mbar_wait(FULL(st1), ((j + 1) / ATP_NST) & 1, a.limit_ns, s_abort)) {
                ok = false;
                break;
              }
              tc_fence_after();
            }
            issue_s(x, st1);
            tc_commit(S_FULL(x));
          } else {
            tc_commit(O_FINAL(x));
          }
        }
      }
      if (!ok) {
        *s_abort = 1;
        report_status(a.status, DECOMOE_ERR_TIMEOUT);
        if (issued) {
          int no_abort = 0;
          tc_commit(DRAIN);
          mbar_wait(DRAIN, 0, a.limit_ns, &no_abort);
        }
      }
    }
  } else {
    // ------------------------------------------------ softmax rows
    const int x = (warp - 2) >> 2;          // head of this warp
    const int q = warp & 3;                 // tensor-memory lane quarter of this warp
    const int r = q * 32 + lane;            // query row of the tile
    const int64_t climit = a.C - 1;
    const int64_t qlim = p0 + r < climit ? p0 + r : climit;                    // last visible key of the row
    const int64_t wlim = p0 + q * 32 < climit ? p0 + q * 32 : climit;          // smallest of the warp's rows
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const float sl2 = a.scale_log2;
    float m = 0.f, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nblk; ++j) {
      if (!__all_sync(0xffffffffu, mbar_wait(S_FULL(x), j & 1, a.limit_ns, s_abort))) {  // warp-uniform loads
        ok = false;
        break;
      }
      tc_fence_after();
      const int64_t key0 = static_cast<int64_t>(j) * ATP_BN;
      uint32_t sv[ATP_BN];
      tmem_ld32(S_TM(x) + lane_off, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
      tmem_ld32(S_TM(x) + lane_off + 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
      tc_wait_ld();
      after_wait(sv);
      if (key0 + ATP_BN - 1 > wlim) {  // the causal edge or the end of the keys crosses this warp's rows
        const int64_t d = qlim - key0;
        const int lim = d < 0 ? -1 : static_cast<int>(d);  // d < 64 here
#pragma unroll
        for (int c = 0; c < ATP_BN; ++c)
          if (c > lim) sv[c] = __float_as_uint(-INFINITY);
      }
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int c = 0; c < ATP_BN; ++c) mx[c & 3] = fmaxf(mx[c & 3], __uint_as_float(sv[c]));
      const float m_blk = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * sl2;
      float factor = 1.0f;
      if (j == 0) {
        m = m_blk;  // key 0 is visible to every row
      } else if (m_blk > m + ATP_RESCALE) {
        factor = ex2_approx(m - m_blk);
        m = m_blk;
        l *= factor;
      }
      if (__any_sync(0xffffffffu, factor != 1.0f)) {
        // the previous product into O has completed (S_FULL is committed after it)
#pragma unroll
        for (int c = 0; c < ATT_D / 32; ++c) {
          uint32_t ov[32];
          tmem_ld32(O_TM(x) + lane_off + 32 * c, ov);
          tc_wait_ld();
          after_wait(ov);
#pragma unroll
          for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * factor);
          tmem_st32(O_TM(x) + lane_off + 32 * c, ov);
        }
      }
      float ls[4] = {0.f, 0.f, 0.f, 0.f};
      uint32_t pk[32];
#pragma unroll
      for (int c = 0; c < ATP_BN; c += 2) {
        const float e0 = ex2_approx(fmaf(__uint_as_float(sv[c]), sl2, -m));
        const float e1 = ex2_approx(fmaf(__uint_as_float(sv[c + 1]), sl2, -m));
        ls[(c >> 1) & 3] += e0 + e1;
        pk[c >> 1] = pack_bf16x2(e0, e1);
      }
      l += (ls[0] + ls[1]) + (ls[2] + ls[3]);
      tmem_st32(P_TM(x) + lane_off, pk);
      tc_wait_st();
      tc_fence_before();
      mbar_arrive(P_FULL(x));
    }
    if (ok && __all_sync(0xffffffffu, mbar_wait(O_FINAL(x), 0, a.limit_ns, s_abort))) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int64_t row = static_cast<int64_t>(qt) * ATP_BM + r;
      uint4* dst = reinterpret_cast<uint4*>(a.out + (row * a.Hq + h0 + x) * ATT_D);
#pragma unroll
      for (int c = 0; c < ATT_D / 32; ++c) {
        uint32_t ov[32];
        tmem_ld32(O_TM(x) + lane_off + 32 * c, ov);
        tc_wait_ld();
        after_wait(ov);
        if (row < a.n) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float* o = reinterpret_cast<const float*>(&ov[8 * u]);
            dst[4 * c + u] = make_uint4(pack_bf16x2(o[0] * inv, o[1] * inv), pack_bf16x2(o[2] * inv, o[3] * inv),
                                        pack_bf16x2(o[4] * inv, o[5] * inv), pack_bf16x2(o[6] * inv, o[7] * inv));
          }
        }
      }
    } else {
      *s_abort = 1;
      report_status(a.status, DECOMOE_ERR_TIMEOUT);
    }
  }
  pdl_trigger();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, ATP_TMEM_COLS);
  }
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

static bool att_use_prefill(int64_t n, int Hq, int Hkv) { return n * (Hq / Hkv) > ATT_MAXQ; }
static int64_t att_c_pad(int64_t C) { return (C + 63) / 64 * 64; }

size_t decomoe_attention_workspace_bytes(int64_t n, int64_t C, int Hq, int Hkv, int D) {
  if (n <= 0 || C <= 0 || Hq <= 0 || Hkv <= 0 || D != ATT_D || Hq % Hkv != 0) return 0;
  if (att_use_prefill(n, Hq, Hkv))  // the transposed values [Hkv][D][C padded to 64]
    return align_up(static_cast<size_t>(Hkv) * ATT_D * att_c_pad(C) * 2, 256);
  const int64_t nsplit = (C + att_chunk(C, Hkv) - 1) / att_chunk(C, Hkv);
  const int64_t nq = n * (Hq / Hkv);
  return align_up(static_cast<size_t>(nsplit) * Hkv * nq * ATT_PROW * sizeof(float), 256);
}

int decomoe_attention(const void* q, int64_t n, const void* k_cache, const void* v_cache, int64_t C, int Hq,
                      int Hkv, int D, float scale, void* out, void* ws, size_t ws_bytes, int32_t* status_dev,
                      decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(D == ATT_D, "attention: head dimension %d (only %d)", D, ATT_D);
  DM_ARG_CHECK(Hq >= 1 && Hkv >= 1 && Hq % Hkv == 0, "attention: Hq=%d must be a multiple of Hkv=%d", Hq, Hkv);
  DM_ARG_CHECK(n >= 0 && C >= n, "attention: need 0 <= n <= C (n=%lld, C=%lld)", (long long)n, (long long)C);
  if (n == 0) return DECOMOE_OK;
  DM_ARG_CHECK(q && k_cache && v_cache && out, "attention: null pointer");
  DM_ARG_CHECK(aligned16(q) && aligned16(k_cache) && aligned16(v_cache) && aligned16(out),
               "attention: pointers must be 16-byte aligned");
  const int G = Hq / Hkv;
  const size_t need = decomoe_attention_workspace_bytes(n, C, Hq, Hkv, D);
  if (ws == nullptr || ws_bytes < need) {
    set_error("attention: workspace needs %zu bytes", need);
    return DECOMOE_ERR_WORKSPACE;
  }
  DM_ARG_CHECK(aligned16(ws), "attention: workspace must be 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const float sc = scale > 0.f ? scale : 1.0f / sqrtf(static_cast<float>(D));
  if (att_use_prefill(n, Hq, Hkv)) {
    DM_ARG_CHECK(G % ATP_HEADS == 0, "attention: prefill sizes need an even number of query heads per KV head (%d)",
                 G);
    // V transposed (keys contiguous) so that P V_j takes K-major operands
    const int64_t C_pad = att_c_pad(C);
    __nv_bfloat16* vt = static_cast<__nv_bfloat16*>(ws);
    DM_CUDA_CHECK(launch_pdl(k_attn_vt, dim3(static_cast<unsigned>(C_pad / 32), ATT_D / 32, Hkv), dim3(256), 0, s,
                             static_cast<const __nv_bfloat16*>(v_cache), C, Hkv, C_pad, vt));
    CUtensorMap tq, tk, tv;
    const uint64_t dq[3] = {static_cast<uint64_t>(D), static_cast<uint64_t>(Hq), static_cast<uint64_t>(n)};
    const uint64_t sq[2] = {static_cast<uint64_t>(D) * 2, static_cast<uint64_t>(Hq) * D * 2};
    const uint64_t dk[3] = {static_cast<uint64_t>(D), static_cast<uint64_t>(Hkv), static_cast<uint64_t>(C)};
    const uint64_t sk[2] = {static_cast<uint64_t>(D) * 2, static_cast<uint64_t>(Hkv) * D * 2};
    const uint64_t dv[3] = {static_cast<uint64_t>(C_pad), static_cast<uint64_t>(D), static_cast<uint64_t>(Hkv)};
    const uint64_t sv[2] = {static_cast<uint64_t>(C_pad) * 2, static_cast<uint64_t>(D) * C_pad * 2};
    const uint32_t bq[3] = {64, 1, ATP_BM}, bk[3] = {64, 1, ATP_BN}, bv[3] = {ATP_BN, ATT_D, 1};
    DM_RET(make_tmap_bf16_3d(&tq, q, dq, sq, bq));
    DM_RET(make_tmap_bf16_3d(&tk, k_cache, dk, sk, bk));
    DM_RET(make_tmap_bf16_3d(&tv, vt, dv, sv, bv));
    AttPreArgs pa;
    pa.n = n;
    pa.C = C;
    pa.Hq = Hq;
    pa.group = G;
    pa.scale_log2 = sc * 1.4426950408889634f;
    pa.out = static_cast<__nv_bfloat16*>(out);
    pa.status = status_dev;
    pa.limit_ns = static_cast<uint64_t>(wait_limit_ns());
    const int64_t ntile = (n + ATP_BM - 1) / ATP_BM;
    DM_ARG_CHECK(ntile * (Hq / ATP_HEADS) < 0x7fffffffLL, "attention: too many query tiles");
    DM_CUDA_CHECK(cudaFuncSetAttribute(k_attn_prefill, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(ATP_SMEM)));
    DM_CUDA_CHECK(launch_pdl(k_attn_prefill, dim3(static_cast<unsigned>(ntile * (Hq / ATP_HEADS))), dim3(ATP_THREADS),
                             ATP_SMEM, s,
                             tq, tk, tv, pa));
    return DECOMOE_OK;
  }
  AttArgs a;
  a.q = static_cast<const uint4*>(q);
  a.k = static_cast<const uint4*>(k_cache);
  a.v = static_cast<const uint4*>(v_cache);
  a.n = n;
  a.C = C;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.chunk = att_chunk(C, Hkv);
  a.nsplit = static_cast<int>((C + a.chunk - 1) / a.chunk);
  DM_ARG_CHECK(a.nsplit <= ATT_MAX_SPLITS, "attention: C=%lld is more than %d keys", (long long)C,
               ATT_MAX_SPLITS * ATT_CH_MAX);
  a.scale = sc;
  a.part = static_cast<float*>(ws);
  const size_t smem = att_split_smem();
  DM_CUDA_CHECK(cudaFuncSetAttribute(k_attn_split, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(smem)));
  DM_CUDA_CHECK(launch_pdl(k_attn_split, dim3(a.nsplit, Hkv), dim3(ATT_THREADS), smem, s, a));
  DM_CUDA_CHECK(launch_pdl(k_attn_combine, dim3(static_cast<unsigned>(n * Hq), ATT_D / 32), dim3(32 * ATT_CWARPS), 0, s,
                           static_cast<const float*>(a.part), n, Hq, Hkv, a.nsplit,
                           static_cast<__nv_bfloat16*>(out)));
  return DECOMOE_OK;
}

}  // extern "C"
