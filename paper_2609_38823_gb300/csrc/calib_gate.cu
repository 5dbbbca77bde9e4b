// Offline RCEP calibration (DecoMoE Section 3.3, Eqs. 8-9; Algorithm 1):
// per-case text-token routed mass, the Mean-Mass expert order and the
// permutation gather that stores experts in that order. And the SAVB exit
// gate (Section 3.2, Eqs. 2-3): pooled text feature, two-class MLP, softmax
// and threshold.
#include "decomoe_internal.cuh"

namespace decomoe {

// ------------------------------------------------------------ calibration

// accum[e] += s[e] / n: the case's routed mass of Eq. 9 (its activated mass
// over n text tokens divided by n), added in call order (one thread per
// expert), so the running sum over cases is reproducible.
__global__ void k_accum_case(const double* __restrict__ s, int E, double n, double* __restrict__ accum) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e < E) accum[e] = __dadd_rn(accum[e], __ddiv_rn(s[e], n));
}

// Eq. 8 on one block: mean[e] = accum[e] / n_cases, and pi lists the experts
// by descending mean, equal means in ascending index (the rank of e counts
// the experts ahead of it). A NaN mean sets DECOMOE_ERR_BAD_INPUT.
__global__ void __launch_bounds__(256)
    k_mean_mass_order(const double* __restrict__ accum, int E, double n_cases, int32_t* __restrict__ pi,
                      double* __restrict__ mean_out, int32_t* status) {
  __shared__ double m[DECOMOE_MAX_E];
  const int e = threadIdx.x;
  double me = 0.0;
  if (e < E) {
    me = __ddiv_rn(accum[e], n_cases);
    m[e] = me;
    if (me != me) report_status(status, DECOMOE_ERR_BAD_INPUT);
  }
  __syncthreads();
  if (e >= E) return;
  int rank = 0;
  for (int j = 0; j < E; ++j) {
    const double mj = m[j];
    rank += (mj > me || (mj == me && j < e)) ? 1 : 0;
  }
  if (rank < E) pi[rank] = e;
  if (mean_out != nullptr) mean_out[e] = me;
}

// dst expert block i = src expert block pi[i]; blockIdx.y = i, blockIdx.x
// strides over the block's 16-byte vectors.
__global__ void __launch_bounds__(256)
    k_permute_vec(const uint4* __restrict__ src, uint4* __restrict__ dst, const int32_t* __restrict__ pi, int E,
                  int64_t nvec, int32_t* status) {
  const int i = blockIdx.y;
  const int from = pi[i];
  if (from < 0 || from >= E) {
    if (blockIdx.x == 0 && threadIdx.x == 0) report_status(status, DECOMOE_ERR_BAD_INPUT);
    return;
  }
  const uint4* s = src + static_cast<int64_t>(from) * nvec;
  uint4* d = dst + static_cast<int64_t>(i) * nvec;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x * 4;
  for (int64_t v = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) * 4; v < nvec; v += stride) {
    uint4 r[4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (v + u < nvec) r[u] = __ldg(s + v + u);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (v + u < nvec) d[v + u] = r[u];
  }
}

// The same for expert blocks whose size is not a multiple of 16 bytes.
__global__ void k_permute_bytes(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                const int32_t* __restrict__ pi, int E, int64_t nbytes, int32_t* status) {
  const int i = blockIdx.y;
  const int from = pi[i];
  if (from < 0 || from >= E) {
    if (blockIdx.x == 0 && threadIdx.x == 0) report_status(status, DECOMOE_ERR_BAD_INPUT);
    return;
  }
  for (int64_t b = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; b < nbytes;
       b += static_cast<int64_t>(gridDim.x) * blockDim.x)
    dst[static_cast<int64_t>(i) * nbytes + b] = src[static_cast<int64_t>(from) * nbytes + b];
}

// ------------------------------------------------------------ SAVB gate

constexpr int GATE_COLS = 64;  // feature columns per pooling block

template <typename T>
struct Vec8;  // eight consecutive elements of a hidden row as fp32
template <>
struct Vec8<__nv_bfloat16> {
  static __device__ __forceinline__ void load(const __nv_bfloat16* p, float (&v)[8]) {
    const uint4 r = __ldg(reinterpret_cast<const uint4*>(p));
    v[0] = bf16_lo(r.x);
    v[1] = bf16_hi(r.x);
    v[2] = bf16_lo(r.y);
    v[3] = bf16_hi(r.y);
    v[4] = bf16_lo(r.z);
    v[5] = bf16_hi(r.z);
    v[6] = bf16_lo(r.w);
    v[7] = bf16_hi(r.w);
  }
};
template <>
struct Vec8<float> {
  static __device__ __forceinline__ void load(const float* p, float (&v)[8]) {
    const float4 a = __ldg(reinterpret_cast<const float4*>(p));
    const float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
};

// Eq. 2: x[c] = mean of text rows 0..n-2 at column c, x[d + c] = text row n-1.
// Text row j is hidden row j, or j + nv from v0 on (the rows outside the
// visual block). Block b owns columns [64b, 64b + 64): thread (r, g) with
// r = tid / 8 sums rows r, r + 32, ... of the eight columns 64b + 8g.. in
// order (fp32), then a fixed tree over r combines the 32 partial sums.
template <typename T>
__global__ void __launch_bounds__(256)
    k_gate_pool(const T* __restrict__ h, int d, int64_t n, int64_t v0, int64_t nv, float* __restrict__ x) {
  __shared__ float red[32][GATE_COLS + 1];
  const int tid = threadIdx.x, r = tid >> 3, g = tid & 7;
  const int c0 = blockIdx.x * GATE_COLS + 8 * g;
  float acc[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = 0.f;
  const int64_t npool = n - 1;
  for (int64_t j = r; j < npool; j += 32) {
    const int64_t row = (j < v0) ? j : j + nv;
    float v[8];
    Vec8<T>::load(h + row * d + c0, v);
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] += v[i];
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) red[r][8 * g + i] = acc[i];
  __syncthreads();
  for (int w = 16; w > 0; w >>= 1) {
    if (r < w) {
#pragma unroll
      for (int i = 0; i < 8; ++i) red[r][8 * g + i] += red[r + w][8 * g + i];
    }
    __syncthreads();
  }
  if (tid < GATE_COLS) {
    const int c = blockIdx.x * GATE_COLS + tid;
    x[c] = (npool > 0) ? red[0][tid] / static_cast<float>(npool) : 0.f;
  } else if (tid < 2 * GATE_COLS && (tid - GATE_COLS) % 8 == 0) {
    const int64_t last = n - 1;
    const int64_t row = (last < v0) ? last : last + nv;
    float v[8];
    const int cc = blockIdx.x * GATE_COLS + (tid - GATE_COLS);
    Vec8<T>::load(h + row * d + cc, v);
#pragma unroll
    for (int i = 0; i < 8; ++i) x[d + cc + i] = v[i];
  }
}

// Eq. 3: hid[u] = relu(W1[u, :] . x + b1[u]), one warp per hidden unit (lanes
// over float4 columns in order, then a shuffle tree). The last block to
// finish (counter) computes z = W2 hid + b2, p_exit = softmax(z)_1 and the
// decision p_exit >= theta.
__global__ void __launch_bounds__(256)
    k_gate_mlp(const float* __restrict__ x, int D2, const float* __restrict__ w1, const float* __restrict__ b1,
               const float* __restrict__ w2, const float* __restrict__ b2, int H, float theta,
               float* __restrict__ hid, unsigned* counter, float* __restrict__ p_exit, int32_t* __restrict__ exit_flag) {
  extern __shared__ float4 xs4[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nv4 = D2 / 4;
  for (int i = tid; i < nv4; i += 256) xs4[i] = reinterpret_cast<const float4*>(x)[i];
  __syncthreads();
  const int u = blockIdx.x * 8 + warp;
  if (u < H) {
    const float4* wr = reinterpret_cast<const float4*>(w1 + static_cast<int64_t>(u) * D2);
    float acc = 0.f;
    for (int i = lane; i < nv4; i += 32) {
      const float4 a = __ldg(wr + i), b = xs4[i];
      acc = fmaf(a.x, b.x, acc);
      acc = fmaf(a.y, b.y, acc);
      acc = fmaf(a.z, b.z, acc);
      acc = fmaf(a.w, b.w, acc);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) hid[u] = fmaxf(acc + b1[u], 0.f);
  }
  __shared__ bool last;
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    last = (atomicAdd(counter, 1u) == gridDim.x - 1);
  }
  __syncthreads();
  if (!last || warp != 0) return;
  __threadfence();
  float z0 = 0.f, z1 = 0.f;
  for (int i = lane; i < H; i += 32) {
    const float hv = __ldcg(hid + i);
    z0 = fmaf(w2[i], hv, z0);
    z1 = fmaf(w2[H + i], hv, z1);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    z0 += __shfl_xor_sync(0xffffffffu, z0, off);
    z1 += __shfl_xor_sync(0xffffffffu, z1, off);
  }
  if (lane == 0) {
    z0 += b2[0];
    z1 += b2[1];
    const float mx = fmaxf(z0, z1);
    const float e0 = __expf(z0 - mx), e1 = __expf(z1 - mx);
    const float p = e1 / (e0 + e1);
    *p_exit = p;
    *exit_flag = (p >= theta) ? 1 : 0;
  }
}

struct CalibLayout {
  size_t part, mass, total;
};
static CalibLayout calib_layout(int64_t T, int E) {
  CalibLayout L;
  const int64_t nb = (T + 7) / 8;
  L.part = 0;
  L.mass = align_up(static_cast<size_t>(nb > 0 ? nb : 1) * E * sizeof(double), 256);
  L.total = align_up(L.mass + static_cast<size_t>(E) * sizeof(double), 256);
  return L;
}

struct GateLayout {
  size_t x, hid, counter, total;
};
static GateLayout gate_layout(int d, int H) {
  GateLayout L;
  L.x = 0;
  L.hid = align_up(static_cast<size_t>(2) * d * sizeof(float), 256);
  L.counter = align_up(L.hid + static_cast<size_t>(H) * sizeof(float), 256);
  L.total = L.counter + 256;
  return L;
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

size_t decomoe_calib_workspace_bytes(int64_t T, int E) {
  if (T < 0 || E <= 0) return 0;
  return calib_layout(T, E).total;
}

int decomoe_calib_case_mass(const float* logits, int64_t T, int E, int64_t ld, int k, int64_t v0, int64_t nv,
                            double* accum, void* ws, size_t ws_bytes, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(E >= 1 && E <= DECOMOE_MAX_E, "calib_case_mass: E=%d outside [1, %d]", E, DECOMOE_MAX_E);
  DM_ARG_CHECK(k >= 1 && k <= DECOMOE_MAX_TOPK && k <= E, "calib_case_mass: bad k=%d", k);
  DM_ARG_CHECK(ld >= E, "calib_case_mass: ld < E");
  DM_ARG_CHECK(v0 >= 0 && nv >= 0 && v0 + nv <= T, "calib_case_mass: visual block [%lld, %lld) outside [0, %lld)",
               (long long)v0, (long long)(v0 + nv), (long long)T);
  const int64_t n = T - nv;
  DM_ARG_CHECK(n >= 1, "calib_case_mass: a case needs at least one text token");
  DM_ARG_CHECK(logits && accum, "calib_case_mass: null pointer");
  const CalibLayout L = calib_layout(n, E);
  if (ws == nullptr || ws_bytes < L.total) {
    set_error("calib_case_mass: workspace needs %zu bytes", L.total);
    return DECOMOE_ERR_WORKSPACE;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint8_t* base = static_cast<uint8_t*>(ws);
  double* part = reinterpret_cast<double*>(base + L.part);
  double* mass = reinterpret_cast<double*>(base + L.mass);
  DM_RET(launch_skip_mass(logits, n, E, ld, k, v0, nv, part, mass, s));
  k_accum_case<<<(E + 255) / 256, 256, 0, s>>>(mass, E, static_cast<double>(n), accum);
  DM_LAUNCH_CHECK("k_accum_case");
  return DECOMOE_OK;
}

int decomoe_mean_mass_order(const double* accum, int E, int n_cases, int32_t* pi, double* mean_out,
                            int32_t* status_dev, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(E >= 1 && E <= DECOMOE_MAX_E, "mean_mass_order: E=%d outside [1, %d]", E, DECOMOE_MAX_E);
  DM_ARG_CHECK(n_cases >= 1, "mean_mass_order: n_cases must be >= 1");
  DM_ARG_CHECK(accum && pi, "mean_mass_order: null pointer");
  k_mean_mass_order<<<1, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(accum, E, static_cast<double>(n_cases), pi,
                                                                          mean_out, status_dev);
  DM_LAUNCH_CHECK("k_mean_mass_order");
  return DECOMOE_OK;
}

int decomoe_permute_experts(const void* src, void* dst, const int32_t* pi, int E, int64_t bytes_per_expert,
                            int32_t* status_dev, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(E >= 1 && E <= 65535, "permute_experts: E=%d outside [1, 65535]", E);
  DM_ARG_CHECK(bytes_per_expert >= 0, "permute_experts: negative size");
  if (bytes_per_expert == 0) return DECOMOE_OK;
  DM_ARG_CHECK(src && dst && pi, "permute_experts: null pointer");
  const uint8_t* s8 = static_cast<const uint8_t*>(src);
  const uint8_t* d8 = static_cast<const uint8_t*>(dst);
  const int64_t total = bytes_per_expert * E;
  DM_ARG_CHECK(d8 + total <= s8 || s8 + total <= d8, "permute_experts: src and dst overlap");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (bytes_per_expert % 16 == 0 && aligned16(src) && aligned16(dst)) {
    const int64_t nvec = bytes_per_expert / 16;
    const int64_t want = (nvec + 1023) / 1024;  // 256 threads x 4 vectors per block
    const int gx = static_cast<int>(std::min<int64_t>(std::max<int64_t>(want, 1), 4096));
    k_permute_vec<<<dim3(gx, E), 256, 0, s>>>(static_cast<const uint4*>(src), static_cast<uint4*>(dst), pi, E, nvec,
                                             status_dev);
    DM_LAUNCH_CHECK("k_permute_vec");
  } else {
    const int64_t want = (bytes_per_expert + 255) / 256;
    const int gx = static_cast<int>(std::min<int64_t>(std::max<int64_t>(want, 1), 4096));
    k_permute_bytes<<<dim3(gx, E), 256, 0, s>>>(static_cast<const uint8_t*>(src), static_cast<uint8_t*>(dst), pi, E,
                                               bytes_per_expert, status_dev);
    DM_LAUNCH_CHECK("k_permute_bytes");
  }
  return DECOMOE_OK;
}

size_t decomoe_savb_gate_workspace_bytes(int d, int H) {
  if (d <= 0 || H <= 0) return 0;
  return gate_layout(d, H).total;
}

int decomoe_savb_gate(const void* h, int64_t T, int d, int dtype, int64_t v0, int64_t nv, const float* w1,
                      const float* b1, const float* w2, const float* b2, int H, float theta, float* p_exit,
                      int32_t* exit_flag, void* ws, size_t ws_bytes, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "savb_gate: bad dtype");
  DM_ARG_CHECK(d > 0 && d % GATE_COLS == 0, "savb_gate: d=%d must be a positive multiple of %d", d, GATE_COLS);
  DM_ARG_CHECK(H >= 1 && H <= (1 << 20), "savb_gate: bad H=%d", H);
  DM_ARG_CHECK(2 * static_cast<int64_t>(d) * 4 <= 200 * 1024, "savb_gate: d=%d too large for the staged feature", d);
  DM_ARG_CHECK(v0 >= 0 && nv >= 0 && v0 + nv <= T, "savb_gate: visual block outside the sequence");
  DM_ARG_CHECK(T - nv >= 1, "savb_gate: no text rows");
  DM_ARG_CHECK(h && w1 && b1 && w2 && b2 && p_exit && exit_flag, "savb_gate: null pointer");
  DM_ARG_CHECK(aligned16(h) && aligned16(w1), "savb_gate: h and w1 must be 16-byte aligned");
  const GateLayout L = gate_layout(d, H);
  if (ws == nullptr || ws_bytes < L.total) {
    set_error("savb_gate: workspace needs %zu bytes", L.total);
    return DECOMOE_ERR_WORKSPACE;
  }
  DM_ARG_CHECK(aligned16(ws), "savb_gate: workspace must be 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint8_t* base = static_cast<uint8_t*>(ws);
  float* x = reinterpret_cast<float*>(base + L.x);
  float* hid = reinterpret_cast<float*>(base + L.hid);
  unsigned* counter = reinterpret_cast<unsigned*>(base + L.counter);
  const int64_t n = T - nv;
  DM_CUDA_CHECK(cudaMemsetAsync(counter, 0, sizeof(unsigned), s));
  if (dtype == DECOMOE_BF16)
    k_gate_pool<__nv_bfloat16><<<d / GATE_COLS, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(h), d, n, v0, nv, x);
  else
    k_gate_pool<float><<<d / GATE_COLS, 256, 0, s>>>(static_cast<const float*>(h), d, n, v0, nv, x);
  DM_LAUNCH_CHECK("k_gate_pool");
  const int D2 = 2 * d;
  const size_t smem = static_cast<size_t>(D2) * sizeof(float);
  if (smem > 48 * 1024)
    DM_CUDA_CHECK(cudaFuncSetAttribute(k_gate_mlp, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)));
  k_gate_mlp<<<(H + 7) / 8, 256, smem, s>>>(x, D2, w1, b1, w2, b2, H, theta, hid, counter, p_exit, exit_flag);
  DM_LAUNCH_CHECK("k_gate_mlp");
  return DECOMOE_OK;
}

}  // extern "C"
