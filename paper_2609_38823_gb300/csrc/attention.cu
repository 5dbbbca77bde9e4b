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

}  // namespace decomoe

using namespace decomoe;

extern "C" {

size_t decomoe_attention_workspace_bytes(int64_t n, int64_t C, int Hq, int Hkv, int D) {
  if (n <= 0 || C <= 0 || Hq <= 0 || Hkv <= 0 || D != ATT_D || Hq % Hkv != 0) return 0;
  const int64_t nsplit = (C + att_chunk(C, Hkv) - 1) / att_chunk(C, Hkv);
  const int64_t nq = n * (Hq / Hkv);
  return align_up(static_cast<size_t>(nsplit) * Hkv * nq * ATT_PROW * sizeof(float), 256);
}

int decomoe_attention(const void* q, int64_t n, const void* k_cache, const void* v_cache, int64_t C, int Hq,
                      int Hkv, int D, float scale, void* out, void* ws, size_t ws_bytes, int32_t* status_dev,
                      decomoe_stream_t stream) {
  clear_error();
  (void)status_dev;
  DM_ARG_CHECK(D == ATT_D, "attention: head dimension %d (only %d)", D, ATT_D);
  DM_ARG_CHECK(Hq >= 1 && Hkv >= 1 && Hq % Hkv == 0, "attention: Hq=%d must be a multiple of Hkv=%d", Hq, Hkv);
  DM_ARG_CHECK(n >= 0 && C >= n, "attention: need 0 <= n <= C (n=%lld, C=%lld)", (long long)n, (long long)C);
  if (n == 0) return DECOMOE_OK;
  DM_ARG_CHECK(q && k_cache && v_cache && out, "attention: null pointer");
  DM_ARG_CHECK(aligned16(q) && aligned16(k_cache) && aligned16(v_cache) && aligned16(out),
               "attention: pointers must be 16-byte aligned");
  const int G = Hq / Hkv;
  DM_ARG_CHECK(n * G <= ATT_MAXQ, "attention: %lld queries per KV head (at most %d in one launch)",
               (long long)(n * G), ATT_MAXQ);
  const size_t need = decomoe_attention_workspace_bytes(n, C, Hq, Hkv, D);
  if (ws == nullptr || ws_bytes < need) {
    set_error("attention: workspace needs %zu bytes", need);
    return DECOMOE_ERR_WORKSPACE;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
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
  a.scale = scale > 0.f ? scale : 1.0f / sqrtf(static_cast<float>(D));
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
