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
// attention on tcgen05. CTA = (query head h, tile of 128 query rows). Per
// block j of 128 keys: S = Q K_j^T (M = 128 queries, N = 128 keys, K = 128
// features) into tensor memory; four warps (one query row per thread) take
// the row's running maximum m and sum l, write p = exp(s - m) as bf16 into a
// 128-byte-swizzled shared-memory tile (the next MMA's A operand) and scale
// their fp32 output row by exp(m_old - m); then O_j = P V_j (N = 128
// features, K = 128 keys, V pre-transposed so both operands are K-major)
// into tensor memory, added to the row in registers. Warp 0 streams K_j and
// V_j^T blocks by TMA into a two-stage ring; warp 1 issues the MMAs. Every
// wait is bounded; on a timeout the CTA records DECOMOE_ERR_TIMEOUT, lets
// its copies and MMAs land, frees its tensor memory and returns.
constexpr int ATP_BM = 128;                 // query rows per CTA
constexpr int ATP_BN = 128;                 // keys per block
constexpr int ATP_HALF = 128 * 64 * 2;      // one 128-row x 64-column swizzled tile (16 KB)
constexpr int ATP_THREADS = 192;
constexpr int ATP_TMEM_COLS = 256;          // S (128 columns) and O_j (128 columns)
constexpr size_t ATP_SMEM = 1024 + 2 * ATP_HALF /* Q */ + 2 * 2 * ATP_HALF /* K ring */ +
                            2 * 2 * ATP_HALF /* V^T ring */ + 2 * ATP_HALF /* P */ + 16 * 8 + 16;

struct AttPreArgs {
  int64_t n, C;        // queries (the last n positions), keys
  int Hq, Hkv;
  float scale;
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

__global__ void __launch_bounds__(ATP_THREADS, 1)
    k_attn_prefill(const __grid_constant__ CUtensorMap tma_q, const __grid_constant__ CUtensorMap tma_k,
                   const __grid_constant__ CUtensorMap tma_vt, const AttPreArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sQ = raw + pad;                 // 2 halves (features 0-63, 64-127)
  const uint32_t sK = sQ + 2 * ATP_HALF;         // [stage][half]
  const uint32_t sV = sK + 4 * ATP_HALF;         // [stage][half of the keys]
  const uint32_t sP = sV + 4 * ATP_HALF;         // [half of the keys]
  uint8_t* pP = smem + (sP - sQ);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 12 * ATP_HALF);
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(bars + 16);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  const uint32_t bar0 = smem_u32(bars);
  const uint32_t Q_BAR = bar0, S_FULL = bar0 + 8, P_FULL = bar0 + 16, O_FULL = bar0 + 24, O_EMPTY = bar0 + 32,
                 DRAIN = bar0 + 40;
  auto FULL = [&](int st) { return bar0 + 48u + 8u * st; };
  auto EMPTY = [&](int st) { return bar0 + 64u + 8u * st; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.Hq / a.Hkv;
  const int ntile = static_cast<int>((a.n + ATP_BM - 1) / ATP_BM);
  // heaviest tiles (most key blocks) first; the heads of a KV group adjacent
  const int h = blockIdx.x % a.Hq;
  const int qt = ntile - 1 - static_cast<int>(blockIdx.x / a.Hq);
  const int g = h / G;
  const int64_t p0 = a.C - a.n + static_cast<int64_t>(qt) * ATP_BM;  // position of the tile's first row
  const int64_t last = p0 + ATP_BM - 1 < a.C - 1 ? p0 + ATP_BM - 1 : a.C - 1;
  const int nblk = static_cast<int>(last / ATP_BN) + 1;  // key blocks any row of the tile can see

  if (threadIdx.x == 0) {
    *s_abort = 0;
    mbar_init(Q_BAR, 1);
    mbar_init(S_FULL, 1);
    mbar_init(P_FULL, 128);
    mbar_init(O_FULL, 1);
    mbar_init(O_EMPTY, 128);
    mbar_init(DRAIN, 1);
    for (int st = 0; st < 2; ++st) {
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
  const uint32_t S_TM = tmem, O_TM = tmem + ATP_BN;
  constexpr uint32_t IDESC = idesc_bf16_f32(ATP_BM, ATP_BN);

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0)
    if (lane == 0) {
      tma_prefetch_desc(&tma_q);
      tma_prefetch_desc(&tma_k);
      tma_prefetch_desc(&tma_vt);
      bool ok = true;
      uint32_t armed = 0, armed_ph = 0;
      mbar_arrive_expect_tx(Q_BAR, 2 * ATP_HALF);
      const int qrow0 = qt * ATP_BM;
      tma_load_3d(sQ, &tma_q, Q_BAR, 0, h, qrow0);
      tma_load_3d(sQ + ATP_HALF, &tma_q, Q_BAR, 64, h, qrow0);
      for (int j = 0; j < nblk; ++j) {
        const int st = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        if (!mbar_wait(EMPTY(st), ph ^ 1u, a.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(FULL(st), 4 * ATP_HALF);
        const int key0 = j * ATP_BN;
        tma_load_3d(sK + (2 * st) * ATP_HALF, &tma_k, FULL(st), 0, g, key0);
        tma_load_3d(sK + (2 * st + 1) * ATP_HALF, &tma_k, FULL(st), 64, g, key0);
        tma_load_3d(sV + (2 * st) * ATP_HALF, &tma_vt, FULL(st), key0, 0, g);
        tma_load_3d(sV + (2 * st + 1) * ATP_HALF, &tma_vt, FULL(st), key0 + 64, 0, g);
        armed |= 1u << st;
        armed_ph = (armed_ph & ~(1u << st)) | (ph << st);
      }
      if (!ok) {
        *s_abort = 1;
        report_status(a.status, DECOMOE_ERR_TIMEOUT);
        int no_abort = 0;
        mbar_wait(Q_BAR, 0, a.limit_ns, &no_abort);
        for (int st = 0; st < 2; ++st)
          if ((armed >> st) & 1u) mbar_wait(FULL(st), (armed_ph >> st) & 1u, a.limit_ns, &no_abort);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (lane 0)
    if (lane == 0) {
      bool ok = mbar_wait(Q_BAR, 0, a.limit_ns, s_abort), issued = false;
      for (int j = 0; ok && j < nblk; ++j) {
        const int st = j & 1;
        if (!mbar_wait(FULL(st), (j >> 1) & 1, a.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // S = Q K_j^T over the 128 features (two 64-column halves)
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint64_t ad = smem_desc_kmajor<64>(sQ + kb * ATP_HALF);
          const uint64_t bd = smem_desc_kmajor<64>(sK + (2 * st + kb) * ATP_HALF);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) tc_mma_f16(S_TM, ad + 2u * kk, bd + 2u * kk, IDESC, (kb | kk) != 0 ? 1u : 0u);
        }
        tc_commit(S_FULL);
        issued = true;
        // O_j = P V_j once the softmax rows have written P and read O_{j-1}
        if (!mbar_wait(P_FULL, j & 1, a.limit_ns, s_abort) ||
            (j > 0 && !mbar_wait(O_EMPTY, (j - 1) & 1, a.limit_ns, s_abort))) {
          ok = false;
          break;
        }
        tc_fence_after();
        fence_proxy_async_smem();  // P came through the generic proxy
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint64_t ad = smem_desc_kmajor<64>(sP + kb * ATP_HALF);
          const uint64_t bd = smem_desc_kmajor<64>(sV + (2 * st + kb) * ATP_HALF);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) tc_mma_f16(O_TM, ad + 2u * kk, bd + 2u * kk, IDESC, (kb | kk) != 0 ? 1u : 0u);
        }
        tc_commit(O_FULL);
        tc_commit(EMPTY(st));
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
    // ------------------------------------------------ softmax and output rows
    const int q = warp & 3;                 // tensor-memory lane quarter of this warp
    const int r = q * 32 + lane;            // query row of the tile
    const int64_t qpos = p0 + r;            // its position
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    float o[ATT_D];
#pragma unroll
    for (int d = 0; d < ATT_D; ++d) o[d] = 0.f;
    float m = -FLT_MAX, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nblk; ++j) {
      if (!__all_sync(0xffffffffu, mbar_wait(S_FULL, j & 1, a.limit_ns, s_abort))) {  // warp-uniform tensor-memory loads
        ok = false;
        break;
      }
      tc_fence_after();
      const int64_t key0 = static_cast<int64_t>(j) * ATP_BN;
      // pass 1: the block's maximum over visible keys
      float bmax = -FLT_MAX;
#pragma unroll
      for (int c = 0; c < ATP_BN / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(S_TM + lane_off + 32 * c, v);
        tc_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int64_t kp = key0 + 32 * c + i;
          if (kp <= qpos && kp < a.C) bmax = fmaxf(bmax, __uint_as_float(v[i]) * a.scale);
        }
      }
      const float m_new = fmaxf(m, bmax);
      const float alpha = m == -FLT_MAX ? 0.f : __expf(m - m_new);
      // pass 2: p = exp(s - m_new) as bf16 into the swizzled P tile, and the sum
      float psum = 0.f;
#pragma unroll
      for (int c = 0; c < ATP_BN / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(S_TM + lane_off + 32 * c, v);
        tc_wait_ld();
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const int64_t kp = key0 + 32 * c + i;
          const float e0 = (kp <= qpos && kp < a.C) ? __expf(__uint_as_float(v[i]) * a.scale - m_new) : 0.f;
          const float e1 = (kp + 1 <= qpos && kp + 1 < a.C) ? __expf(__uint_as_float(v[i + 1]) * a.scale - m_new) : 0.f;
          psum += e0 + e1;
          pk[i / 2] = pack_bf16x2(e0, e1);
        }
        // columns 32c .. 32c + 31: half kb = c / 2, 16-byte chunks (c % 2) * 4 .. + 3
        const int kb = c >> 1;
        uint8_t* rowp = pP + kb * ATP_HALF + r * 128;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int chunk = (c & 1) * 4 + u;
          *reinterpret_cast<uint4*>(rowp + ((chunk ^ (r & 7)) << 4)) =
              make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
        }
      }
      l = l * alpha + psum;
      m = m_new;
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(P_FULL);
      if (!__all_sync(0xffffffffu, mbar_wait(O_FULL, j & 1, a.limit_ns, s_abort))) {
        ok = false;
        break;
      }
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < ATT_D / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(O_TM + lane_off + 32 * c, v);
        tc_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) o[32 * c + i] = fmaf(o[32 * c + i], alpha, __uint_as_float(v[i]));
      }
      tc_fence_before();
      mbar_arrive(O_EMPTY);
    }
    if (!ok) {
      *s_abort = 1;
      report_status(a.status, DECOMOE_ERR_TIMEOUT);
    } else if (qt * ATP_BM + r < a.n) {
      const float inv = 1.0f / l;
      uint4* dst = reinterpret_cast<uint4*>(a.out + ((static_cast<int64_t>(qt) * ATP_BM + r) * a.Hq + h) * ATT_D);
#pragma unroll
      for (int c = 0; c < ATT_D / 8; ++c)
        dst[c] = make_uint4(pack_bf16x2(o[8 * c] * inv, o[8 * c + 1] * inv), pack_bf16x2(o[8 * c + 2] * inv, o[8 * c + 3] * inv),
                            pack_bf16x2(o[8 * c + 4] * inv, o[8 * c + 5] * inv), pack_bf16x2(o[8 * c + 6] * inv, o[8 * c + 7] * inv));
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
    const uint32_t bq[3] = {64, 1, ATP_BM}, bk[3] = {64, 1, ATP_BN}, bv[3] = {64, ATT_D, 1};
    DM_RET(make_tmap_bf16_3d(&tq, q, dq, sq, bq));
    DM_RET(make_tmap_bf16_3d(&tk, k_cache, dk, sk, bk));
    DM_RET(make_tmap_bf16_3d(&tv, vt, dv, sv, bv));
    AttPreArgs pa;
    pa.n = n;
    pa.C = C;
    pa.Hq = Hq;
    pa.Hkv = Hkv;
    pa.scale = sc;
    pa.out = static_cast<__nv_bfloat16*>(out);
    pa.status = status_dev;
    pa.limit_ns = static_cast<uint64_t>(wait_limit_ns());
    const int64_t ntile = (n + ATP_BM - 1) / ATP_BM;
    DM_ARG_CHECK(ntile * Hq < 0x7fffffffLL, "attention: too many query tiles");
    DM_CUDA_CHECK(cudaFuncSetAttribute(k_attn_prefill, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(ATP_SMEM)));
    DM_CUDA_CHECK(launch_pdl(k_attn_prefill, dim3(static_cast<unsigned>(ntile * Hq)), dim3(ATP_THREADS), ATP_SMEM, s,
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
