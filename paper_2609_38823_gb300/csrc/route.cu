// Router logits (CUDA-core path) and prefix-restricted top-k routing with the
// activated-mass reduction of RCEP (DecoMoE Section 3.3, Eqs. 10-12,
// Algorithm 2).
#include <cfloat>
#include <cstdint>

#include "dispatch_tile.cuh"
#include "route_common.cuh"

namespace decomoe {

// ------------------------------------------------------------ router, CUDA cores
// logits[t, e] = sum_j x[t, j] * w_r[e, j] + bias[e]. One thread per (t, e);
// fp32 accumulate. Used for fp32 storage and shapes the tensor-core kernel does
// not take.
template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__global__ void k_router_simt(const T* __restrict__ x, const T* __restrict__ w_r,
                              const float* __restrict__ bias, int64_t Tn, int d, int E,
                              float* __restrict__ logits) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= Tn * E) return;
  const int64_t t = i / E;
  const int e = static_cast<int>(i - t * E);
  const T* xr = x + t * d;
  const T* wr = w_r + static_cast<int64_t>(e) * d;
  float acc = 0.f;
  for (int j = 0; j < d; ++j) acc = fmaf(to_f(xr[j]), to_f(wr[j]), acc);
  if (bias != nullptr) acc += bias[e];
  logits[i] = acc;
}

// Router for few tokens (decode) on CUDA cores: fp32 dot products of the bf16
// router rows and token rows. The router matrix is read from HBM once and
// spread over many SMs instead of one tensor-core tile.
#ifndef DECOMOE_ROUTER_GEMV_MAX_T
#define DECOMOE_ROUTER_GEMV_MAX_T 6  // token counts up to which the router runs on CUDA cores
#endif
static constexpr int64_t router_gemv_max_t() { return DECOMOE_ROUTER_GEMV_MAX_T; }
// One block per expert row and GEMV_TPB tokens: the block's 128 threads split
// the row's 16-byte vectors (thread i takes vectors i, i + 128, ...), so a
// row's loads are spread over four warps and the E rows over E blocks (one per
// SM at decode sizes) instead of piling every row of a block onto one SM; all
// of a thread's loads are issued before its first multiply. Partial dots are
// reduced by warp shuffles, then over the four warps in a fixed order.
__global__ void __launch_bounds__(GEMV_THREADS)
    k_router_gemv(const uint4* __restrict__ x, const uint4* __restrict__ w_r, const float* __restrict__ bias,
                  int64_t Tn, int vpr, int E, float* __restrict__ logits) {
  pdl_enter();
  __shared__ float red[GEMV_THREADS / 32][GEMV_TPB];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int e = blockIdx.x;
  const int64_t t0 = static_cast<int64_t>(blockIdx.y) * GEMV_TPB;
  const int nt = Tn - t0 < GEMV_TPB ? static_cast<int>(Tn - t0) : GEMV_TPB;
  const uint4* wr = w_r + static_cast<int64_t>(e) * vpr;
  float acc[GEMV_TPB];
#pragma unroll
  for (int j = 0; j < GEMV_TPB; ++j) acc[j] = 0.f;
  const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
  for (int c0 = 0; c0 < vpr; c0 += GEMV_THREADS * GEMV_VPT) {
    uint4 wv[GEMV_VPT], xv[GEMV_TPB][GEMV_VPT];
#pragma unroll
    for (int i = 0; i < GEMV_VPT; ++i) {
      const int c = c0 + static_cast<int>(threadIdx.x) + GEMV_THREADS * i;
      wv[i] = (c < vpr) ? __ldg(wr + c) : zero;
#pragma unroll
      for (int j = 0; j < GEMV_TPB; ++j) xv[j][i] = (c < vpr && j < nt) ? __ldg(x + (t0 + j) * vpr + c) : zero;
    }
#pragma unroll
    for (int i = 0; i < GEMV_VPT; ++i)
#pragma unroll
      for (int j = 0; j < GEMV_TPB; ++j) acc[j] = dot8_bf16(wv[i], xv[j][i], acc[j]);
  }
#pragma unroll
  for (int j = 0; j < GEMV_TPB; ++j) {
    float v = acc[j];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == 0) red[warp][j] = v;
  }
  __syncthreads();
  if (static_cast<int>(threadIdx.x) < nt) {
    const int j = threadIdx.x;
    float v = red[0][j];
#pragma unroll
    for (int w = 1; w < GEMV_THREADS / 32; ++w) v += red[w][j];
    logits[(t0 + j) * E + e] = v + (bias != nullptr ? bias[e] : 0.f);
  }
}

// ------------------------------------------------------------ routing
// One warp per token; lane l holds logits l, l+32, ... (E <= 256, 8 per lane)
// in registers. A pass of k rounds of warp arg-max picks the k largest of a
// range (ties: lower expert index); pick j ends in lane j. Weights are the
// softmax over the k picks (equal to prefix softmax + top-k + renormalise,
// because the prefix denominator cancels).
//
// With a mass buffer the same launch also computes the activated mass of
// Eq. 11 over the full pool [0, E): the full-pool picks are found first; if
// they all lie inside [0, K) they are also the prefix picks, else a second
// pass runs over [0, K). Each block writes its tokens' fp32 full-pool weights
// per expert, summed in token order, to part[block][e]; k_mass_finalize sums
// the blocks in a fixed order in fp64, so the mass is bit-reproducible.
constexpr int ROUTE_THREADS = 256;
constexpr int ROUTE_TPB = ROUTE_TOKENS_PER_BLOCK;  // tokens per block: one per warp

// NP: 1 reads plain logit rows; NP > 1 reads NP k slices of the split
// router (src), each warp loading its row's slices as coalesced 16-byte
// vectors (all NP in flight), adding them in slice order and the bias last,
// storing the sums to src.logits_out and, through shared memory, into the
// key layout (E % 4 == 0, 16-byte aligned rows).
// rd.counts set (one block, T <= ROUTE_TPB): after routing, the block
// dispatches its own picks (dispatch_tile over the T*k pairs).
static_assert(ROUTE_THREADS == DSP_THREADS, "the routing block runs the dispatch tile");
template <int NP>
__global__ void __launch_bounds__(ROUTE_THREADS)
    k_route(const float* __restrict__ logits, int64_t Tn, int E, int64_t ld, int K, int k,
            int32_t* __restrict__ idx_out, float* __restrict__ w_out, double* __restrict__ part,
            const int32_t* __restrict__ K_dev, int64_t skip_at, int64_t skip_len, RouteSrc src, RouteDispatch rd,
            int32_t* __restrict__ zero_ints, int n_zero) {
  pdl_enter();
  // block 0 clears a small int array for a later launch of the caller's chain
  if (zero_ints != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < n_zero; i += ROUTE_THREADS) zero_ints[i] = 0;
  if (K_dev != nullptr) K = *K_dev;  // prefix chosen on the device (k <= K <= E by construction)
  __shared__ int s_idx[ROUTE_TPB][DECOMOE_MAX_TOPK];
  __shared__ float s_w[ROUTE_TPB][DECOMOE_MAX_TOPK];
  __shared__ float s_row[NP > 1 ? ROUTE_TPB : 1][NP > 1 ? DECOMOE_MAX_E : 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t t = static_cast<int64_t>(blockIdx.x) * ROUTE_TPB + warp;
  const bool mass = part != nullptr;
  if (t < Tn) {
    // token t reads logit row t, or t + skip_len from skip_at on (the text
    // tokens around a removed visual block)
    const int64_t roff = (t < skip_at ? t : t + skip_len) * ld;
    const float* row = logits + roff;
    const int lim = mass ? E : K;
    uint32_t v[8];  // order-preserving keys of the row's logits
    if constexpr (NP == 1) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int e = lane + 32 * i;
        v[i] = (e < lim) ? fkey(row[e]) : 0u;
      }
    } else {
      // partial sums of the k-split router, added in slice order, bias last
      const float4* r4 = reinterpret_cast<const float4*>(row);
      const int64_t s4 = src.part_stride / 4;
      for (int c = lane; c < E / 4; c += 32) {
        float4 p[NP];
#pragma unroll
        for (int sl = 0; sl < NP; ++sl) p[sl] = __ldcs(r4 + sl * s4 + c);
        float4 a = p[0];
#pragma unroll
        for (int sl = 1; sl < NP; ++sl) {
          a.x += p[sl].x;
          a.y += p[sl].y;
          a.z += p[sl].z;
          a.w += p[sl].w;
        }
        if (src.bias != nullptr) {
          const float4 b = reinterpret_cast<const float4*>(src.bias)[c];
          a.x += b.x;
          a.y += b.y;
          a.z += b.z;
          a.w += b.w;
        }
        if (src.logits_out != nullptr) reinterpret_cast<float4*>(src.logits_out + roff)[c] = a;
        reinterpret_cast<float4*>(s_row[warp])[c] = a;
      }
      __syncwarp();
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int e = lane + 32 * i;
        v[i] = (e < lim) ? fkey(s_row[warp][e]) : 0u;
      }
    }
    float my_v;
    int my_i;
    warp_topk(v, lim, k, lane, my_v, my_i);
    if (mass) {
      const float wf = pick_weight(my_v, lane, k);
      if (lane < k) {
        s_idx[warp][lane] = my_i;
        s_w[warp][lane] = wf;
      }
      // full-pool picks all inside the prefix: they are the prefix picks too
      const bool inside = __all_sync(0xffffffffu, lane >= k || my_i < K);
      if (!inside) warp_topk(v, K, k, lane, my_v, my_i);
    }
    if (idx_out != nullptr || w_out != nullptr) {
      const float w = pick_weight(my_v, lane, k);
      if (lane < k) {
        if (idx_out != nullptr) idx_out[t * k + lane] = my_i;
        if (w_out != nullptr) w_out[t * k + lane] = w;
      }
    }
  }
  if (mass) {
    __syncthreads();
    const int ntok = static_cast<int>(Tn - static_cast<int64_t>(blockIdx.x) * ROUTE_TPB < ROUTE_TPB
                                          ? Tn - static_cast<int64_t>(blockIdx.x) * ROUTE_TPB
                                          : ROUTE_TPB);
    for (int e = threadIdx.x; e < E; e += ROUTE_THREADS) {
      float acc = 0.f;
      for (int tt = 0; tt < ntok; ++tt)
        for (int j = 0; j < k; ++j)
          if (s_idx[tt][j] == e) acc += s_w[tt][j];  // token order, then slot order
      part[static_cast<int64_t>(blockIdx.x) * E + e] = static_cast<double>(acc);
    }
  }
  if (rd.counts != nullptr) {
    __syncthreads();  // the block's picks in idx_out are visible to all its threads
    dispatch_tile<true>(idx_out, Tn * k, k, rd.Kd, nullptr, 1, 0, rd.counts, rd.offsets, rd.perm_token, rd.inv_slot,
                        rd.status, static_cast<const uint4*>(rd.x), rd.row_vec, static_cast<uint4*>(rd.x_perm));
  }
}

// mass[e] = sum over blocks of part[b][e]: one block per expert, each thread
// sums a fixed strided subset of blocks in order, then a fixed-shape tree in
// shared memory combines the 256 thread sums (bit-reproducible).
__global__ void __launch_bounds__(256)
    k_mass_finalize(const double* __restrict__ part, int nblocks, int E, double* __restrict__ mass) {
  pdl_enter();
  mass_finalize_block(part, nblocks, E, static_cast<int>(blockIdx.x), mass);
}

// Eq. 12 on the device, one thread (bit-identical to decomoe_select_prefix).
__global__ void k_select_prefix(const double* __restrict__ mass, int E, int k, double p, int32_t* __restrict__ K_dev) {
  pdl_enter();
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  *K_dev = select_prefix_seq(mass, E, k, p);
}

// Activated mass (Eq. 11) over n tokens whose logit rows skip a block:
// token t reads row t, or t + skip_len from skip_at on. part needs
// ceil(n / ROUTE_TPB) * E doubles.
int launch_skip_mass(const float* logits, int64_t n, int E, int64_t ld, int k, int64_t skip_at, int64_t skip_len,
                     double* part, double* mass, cudaStream_t s) {
  const int64_t nblocks = (n + ROUTE_TPB - 1) / ROUTE_TPB;
  k_route<1><<<static_cast<unsigned>(nblocks), ROUTE_THREADS, 0, s>>>(logits, n, E, ld, E, k, nullptr, nullptr, part,
                                                                      nullptr, skip_at, skip_len, RouteSrc{},
                                                                      RouteDispatch{}, nullptr, 0);
  DM_LAUNCH_CHECK("k_route");
  k_mass_finalize<<<E, 256, 0, s>>>(part, static_cast<int>(nblocks), E, mass);
  DM_LAUNCH_CHECK("k_mass_finalize");
  return DECOMOE_OK;
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

int decomoe_router_logits(const void* x, const void* w_r, const float* bias, int64_t T, int d,
                          int E, int dtype, float* logits, int32_t* status_dev,
                          decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(T >= 0 && d > 0 && E > 0, "router_logits: bad sizes T=%lld d=%d E=%d", (long long)T, d, E);
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "router_logits: bad dtype %d", dtype);
  if (T == 0) return DECOMOE_OK;
  DM_ARG_CHECK(x && w_r && logits, "router_logits: null pointer");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (dtype == DECOMOE_BF16 && T <= router_gemv_max_t() && d % 8 == 0 && aligned16(x) && aligned16(w_r)) {
    const dim3 grid(static_cast<unsigned>(E), static_cast<unsigned>((T + GEMV_TPB - 1) / GEMV_TPB));
    DM_CUDA_CHECK(launch_pdl(k_router_gemv, grid, dim3(GEMV_THREADS), 0, s, static_cast<const uint4*>(x),
                             static_cast<const uint4*>(w_r), bias, static_cast<int64_t>(T), d / 8, E, logits));
    return DECOMOE_OK;
  }
  if (dtype == DECOMOE_BF16 && router_tc_supported(d, E)) {
    DM_ARG_CHECK(aligned16(x) && aligned16(w_r) && aligned16(logits),
                 "router_logits: pointers must be 16-byte aligned");
    return launch_router_tc(x, w_r, bias, T, d, E, logits, status_dev, s);
  }
  const int64_t n = T * E;
  const int threads = 256;
  const int64_t blocks = (n + threads - 1) / threads;
  if (dtype == DECOMOE_F32)
    k_router_simt<float><<<blocks, threads, 0, s>>>(static_cast<const float*>(x),
                                                    static_cast<const float*>(w_r), bias, T, d, E, logits);
  else
    k_router_simt<__nv_bfloat16><<<blocks, threads, 0, s>>>(
        static_cast<const __nv_bfloat16*>(x), static_cast<const __nv_bfloat16*>(w_r), bias, T, d, E, logits);
  DM_LAUNCH_CHECK("k_router_simt");
  return DECOMOE_OK;
}

size_t decomoe_router_logits_ws_bytes(int64_t T, int d, int E) {
  if (T <= 0 || d <= 0 || E <= 0) return 0;
  if (T <= router_gemv_max_t()) return 0;
  const int ks = router_split_ks(T, d, E);
  return ks > 1 ? align_up(static_cast<size_t>(ks) * T * E * sizeof(float), 256) : 0;
}

int decomoe_router_logits_ws(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E, int dtype,
                             float* logits, void* ws, size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream) {
  clear_error();
  const size_t need = decomoe_router_logits_ws_bytes(T, d, E);
  if (dtype != DECOMOE_BF16 || need == 0 || T <= router_gemv_max_t())
    return decomoe_router_logits(x, w_r, bias, T, d, E, dtype, logits, status_dev, stream);
  DM_ARG_CHECK(x && w_r && logits, "router_logits_ws: null pointer");
  DM_ARG_CHECK(aligned16(x) && aligned16(w_r) && aligned16(logits) && aligned16(ws),
               "router_logits_ws: pointers must be 16-byte aligned");
  if (ws == nullptr || ws_bytes < need) {
    set_error("router_logits_ws: workspace needs %zu bytes", need);
    return DECOMOE_ERR_WORKSPACE;
  }
  return launch_router_split(x, w_r, bias, T, d, E, logits, static_cast<float*>(ws), status_dev,
                             reinterpret_cast<cudaStream_t>(stream));
}

size_t decomoe_route_workspace_bytes(int64_t T, int E) {
  if (T < 0 || E <= 0) return 0;
  const int64_t nblocks = (T + ROUTE_TPB - 1) / ROUTE_TPB;
  return align_up(static_cast<size_t>(nblocks > 0 ? nblocks : 1) * E * sizeof(double), 256);
}

int decomoe_route_prefix(const float* logits, int64_t T, int E, int64_t ld, int K, int k,
                         int32_t* topk_idx, float* topk_w, double* mass_out, void* ws,
                         size_t ws_bytes, decomoe_stream_t stream) {
  clear_error();
  return route_prefix_src(logits, RouteSrc{}, T, E, ld, K, k, topk_idx, topk_w, mass_out, ws, ws_bytes, false,
                          nullptr, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"

namespace decomoe {

int route_prefix_src(const float* logits, const RouteSrc& src, int64_t T, int E, int64_t ld, int K, int k,
                     int32_t* topk_idx, float* topk_w, double* mass_out, void* ws, size_t ws_bytes,
                     bool defer_finalize, int* mass_blocks, cudaStream_t s, const int32_t* K_dev,
                     const RouteDispatch* rd, int32_t* zero_ints, int n_zero) {
  if (mass_blocks != nullptr) *mass_blocks = 0;
  DM_ARG_CHECK(T >= 0, "route_prefix: T < 0");
  DM_ARG_CHECK(E >= 1 && E <= DECOMOE_MAX_E, "route_prefix: E=%d outside [1, %d]", E, DECOMOE_MAX_E);
  DM_ARG_CHECK(k >= 1 && k <= DECOMOE_MAX_TOPK, "route_prefix: k=%d outside [1, %d]", k, DECOMOE_MAX_TOPK);
  DM_ARG_CHECK(K_dev != nullptr || (K >= k && K <= E), "route_prefix: need k <= K <= E (k=%d K=%d E=%d)", k, K, E);
  DM_ARG_CHECK(K_dev == nullptr || mass_out == nullptr, "route_prefix: a device prefix takes no mass");
  DM_ARG_CHECK(ld >= E, "route_prefix: ld < E");
  DM_ARG_CHECK(src.nparts == 1 || ((src.nparts == 4 || src.nparts == 16) && E % 4 == 0 && ld == E &&
                                    src.part_stride % 4 == 0 && aligned16(logits) &&
                                    (src.bias == nullptr || aligned16(src.bias)) &&
                                    (src.logits_out == nullptr || aligned16(src.logits_out))),
               "route_prefix: logit slices need 4 or 16 slices of 16-byte aligned rows");
  if (T == 0) {
    if (mass_out) DM_CUDA_CHECK(cudaMemsetAsync(mass_out, 0, sizeof(double) * E, s));
    return DECOMOE_OK;
  }
  DM_ARG_CHECK(logits != nullptr, "route_prefix: logits is null");
  const int64_t nblocks = (T + ROUTE_TPB - 1) / ROUTE_TPB;
  DM_ARG_CHECK(nblocks <= 0x7fffffff, "route_prefix: T too large");
  double* part = nullptr;
  if (mass_out != nullptr) {
    if (ws == nullptr || ws_bytes < decomoe_route_workspace_bytes(T, E)) {
      set_error("route_prefix: workspace needs %zu bytes", decomoe_route_workspace_bytes(T, E));
      return DECOMOE_ERR_WORKSPACE;
    }
    // one routing block: its partial is the mass itself (the fixed-order
    // finalize would only add zeros), so it is written in place
    part = nblocks == 1 ? mass_out : static_cast<double*>(ws);
  }
  RouteDispatch rdv;
  if (rd != nullptr && rd->counts != nullptr) {
    DM_ARG_CHECK(nblocks == 1 && topk_idx != nullptr && T * k <= DSP_TILE,
                 "route_prefix: dispatch in the routing block needs T <= %d", ROUTE_TPB);
    rdv = *rd;
  }
  auto kern = src.nparts == 16 ? k_route<16> : src.nparts == 4 ? k_route<4> : k_route<1>;
  DM_CUDA_CHECK(launch_pdl(kern, dim3(static_cast<unsigned>(nblocks)), dim3(ROUTE_THREADS), 0, s, logits, T, E, ld,
                           K, k, topk_idx, topk_w, part, K_dev, INT64_MAX, static_cast<int64_t>(0), src, rdv,
                           zero_ints, n_zero));
  if (mass_out != nullptr && nblocks > 1) {
    if (defer_finalize && mass_blocks != nullptr) {
      *mass_blocks = static_cast<int>(nblocks);  // the caller's next kernel adds the partials up
    } else {
      DM_CUDA_CHECK(launch_pdl(k_mass_finalize, dim3(E), dim3(256), 0, s, static_cast<const double*>(part),
                               static_cast<int>(nblocks), E, mass_out));
    }
  }
  return DECOMOE_OK;
}

}  // namespace decomoe

extern "C" {


int decomoe_select_prefix_device(const double* mass, int E, int k, double p, int32_t* K_dev,
                                 decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(mass && K_dev, "select_prefix_device: null pointer");
  DM_ARG_CHECK(E >= 1 && k >= 1 && k <= E, "select_prefix_device: need 1 <= k <= E");
  DM_ARG_CHECK(p > 0.0 && p <= 1.0, "select_prefix_device: p must lie in (0, 1]");
  DM_CUDA_CHECK(launch_pdl(k_select_prefix, dim3(1), dim3(32), 0, reinterpret_cast<cudaStream_t>(stream), mass, E, k,
                           p, K_dev));
  return DECOMOE_OK;
}

int decomoe_route_prefix_dk(const float* logits, int64_t T, int E, int64_t ld, const int32_t* K_dev, int k,
                            int32_t* topk_idx, float* topk_w, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(T >= 0 && E >= 1 && E <= DECOMOE_MAX_E && k >= 1 && k <= DECOMOE_MAX_TOPK && k <= E && ld >= E,
               "route_prefix_dk: bad sizes");
  if (T == 0) return DECOMOE_OK;
  DM_ARG_CHECK(logits && K_dev, "route_prefix_dk: null pointer");
  return route_prefix_src(logits, RouteSrc{}, T, E, ld, E, k, topk_idx, topk_w, nullptr, nullptr, 0, false, nullptr,
                          reinterpret_cast<cudaStream_t>(stream), K_dev);
}

}  // extern "C"
