// Dispatch of the routed (token, slot) pairs to the prefix experts: per-tile
// histograms with warp-aggregated shared-memory atomics, a scan, a stable
// rank assignment, and a 128-bit row gather (DecoMoE Algorithm 2: only the
// first K expert MLPs are evaluated, each on the tokens routed to it).
#include <mutex>

#include "dispatch_tile.cuh"

namespace decomoe {

// Deferred activated mass (Eq. 11) carried by a dispatch launch: blocks
// [first, first + E) of the grid add up the routing blocks' partial masses,
// one expert each, in the fixed order of mass_finalize_block.
struct MassFinish {
  const double* part = nullptr;  // null: nothing to finish
  int nblocks = 0;
  int E = 0;
  double* mass = nullptr;
};

// Pass 1: histogram of expert ids in each tile of DSP_TILE consecutive pairs
// (blocks [0, ntiles)); blocks from ntiles on finish a deferred mass.
__global__ void __launch_bounds__(DSP_THREADS)
    k_dispatch_hist(const int32_t* __restrict__ idx, int64_t N, int K,
                    int32_t* __restrict__ tile_hist, int32_t* status, int ntiles, MassFinish mf) {
  pdl_enter();
  if (static_cast<int>(blockIdx.x) >= ntiles) {
    mass_finalize_block(mf.part, mf.nblocks, mf.E, static_cast<int>(blockIdx.x) - ntiles, mf.mass);
    return;
  }
  __shared__ int hist[DECOMOE_MAX_E];
  for (int e = threadIdx.x; e < K; e += DSP_THREADS) hist[e] = 0;
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t base = static_cast<int64_t>(blockIdx.x) * DSP_TILE + warp * DSP_PER_WARP;
#pragma unroll
  for (int r = 0; r < DSP_PER_WARP / 32; ++r) {
    const int64_t f = base + r * 32 + lane;
    int e = -2;
    if (f < N) {
      e = idx[f];
      if (e < 0 || e >= K) {
        report_status(status, DECOMOE_ERR_BAD_INPUT);
        e = -1;
      }
    }
    const uint32_t grp = __match_any_sync(0xffffffffu, e);
    if (e >= 0 && lane == __ffs(grp) - 1) atomicAdd(&hist[e], __popc(grp));
  }
  __syncthreads();
  for (int e = threadIdx.x; e < K; e += DSP_THREADS)
    tile_hist[static_cast<int64_t>(blockIdx.x) * K + e] = hist[e];
}

// Pass 2: the tile kernel (dispatch_tile). SINGLE: one tile in one block
// (decode sizes); blocks from 1 on finish a deferred mass.
template <bool SINGLE>
__global__ void __launch_bounds__(DSP_THREADS)
    k_dispatch_scatter(const int32_t* __restrict__ idx, int64_t N, int k, int K,
                       const int32_t* __restrict__ tile_hist, int ntiles,
                       int32_t* __restrict__ counts, int32_t* __restrict__ offsets,
                       int32_t* __restrict__ perm_token, int32_t* __restrict__ inv_slot,
                       int32_t* status = nullptr, const uint4* __restrict__ x = nullptr, int row_vec = 0,
                       uint4* __restrict__ x_perm = nullptr, MassFinish mf = MassFinish{}) {
  pdl_enter();
  if (SINGLE && blockIdx.x > 0) {
    mass_finalize_block(mf.part, mf.nblocks, mf.E, static_cast<int>(blockIdx.x) - 1, mf.mass);
    return;
  }
  dispatch_tile<SINGLE>(idx, N, k, K, tile_hist, ntiles, static_cast<int>(blockIdx.x), counts, offsets, perm_token,
                        inv_slot, status, x, row_vec, x_perm);
}

// Pass 3: x_perm[r, :] = x[perm_token[r], :], one warp per row, 16-byte
// vectors, loads of a row issued before its stores.
__global__ void __launch_bounds__(256)
    k_gather_rows(const uint4* __restrict__ x, const int32_t* __restrict__ perm_token,
                  const int32_t* __restrict__ offsets, int K, int vec_per_row,
                  uint4* __restrict__ x_perm) {
  pdl_enter();
  const int rows = offsets[K];
  const int lane = threadIdx.x & 31;
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  for (int r = gw; r < rows; r += nw) {
    const int t = perm_token[r];
    const uint4* src = x + static_cast<int64_t>(t) * vec_per_row;
    uint4* dst = x_perm + static_cast<int64_t>(r) * vec_per_row;
    int c = lane;
    for (; c + 32 * 7 < vec_per_row; c += 32 * 8) {
      uint4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldg(src + c + 32 * u);
#pragma unroll
      for (int u = 0; u < 8; ++u) dst[c + 32 * u] = v[u];
    }
    for (; c < vec_per_row; c += 32) dst[c] = __ldg(src + c);
  }
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

size_t decomoe_dispatch_workspace_bytes(int64_t T, int k, int K) {
  if (T < 0 || k <= 0 || K <= 0) return 0;
  const int64_t N = T * k;
  const int64_t ntiles = (N + DSP_TILE - 1) / DSP_TILE;
  return align_up(static_cast<size_t>(ntiles > 0 ? ntiles : 1) * K * sizeof(int32_t), 256);
}

int decomoe_gather_rows(const void* x, const int32_t* perm_token, const int32_t* offsets, int K, int64_t N,
                        int d, int dtype, void* x_perm, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(N >= 0 && K >= 1 && d > 0 && (dtype == DECOMOE_BF16 || dtype == DECOMOE_F32),
               "gather_rows: bad sizes or dtype");
  if (N == 0) return DECOMOE_OK;
  const size_t row_bytes = static_cast<size_t>(d) * dtype_bytes(dtype);
  DM_ARG_CHECK(x && perm_token && offsets && x_perm, "gather_rows: null pointer");
  DM_ARG_CHECK(row_bytes % 16 == 0 && aligned16(x) && aligned16(x_perm),
               "gather_rows: rows must be 16-byte multiples and 16-byte aligned");
  return launch_gather_rows(x, perm_token, offsets, K, row_bytes, N, x_perm, reinterpret_cast<cudaStream_t>(stream));
}

int decomoe_dispatch(const int32_t* topk_idx, int64_t T, int k, int K, const void* x, int d,
                     int dtype, int32_t* counts, int32_t* offsets, int32_t* perm_token,
                     int32_t* inv_slot, void* x_perm, void* ws, size_t ws_bytes,
                     int32_t* status_dev, decomoe_stream_t stream) {
  clear_error();
  return dispatch_with_mass(topk_idx, T, k, K, x, d, dtype, counts, offsets, perm_token, inv_slot, x_perm, ws,
                            ws_bytes, status_dev, nullptr, 0, 0, nullptr, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"

namespace decomoe {

int dispatch_with_mass(const int32_t* topk_idx, int64_t T, int k, int K, const void* x, int d, int dtype,
                       int32_t* counts, int32_t* offsets, int32_t* perm_token, int32_t* inv_slot, void* x_perm,
                       void* ws, size_t ws_bytes, int32_t* status_dev, const double* mass_part, int mass_blocks,
                       int mass_E, double* mass, cudaStream_t s) {
  MassFinish mf;
  if (mass_part != nullptr && mass_blocks > 0) {
    DM_ARG_CHECK(mass != nullptr && mass_E >= 1 && mass_E <= DECOMOE_MAX_E, "dispatch: bad deferred mass");
    mf.part = mass_part;
    mf.nblocks = mass_blocks;
    mf.E = mass_E;
    mf.mass = mass;
  }
  const int mblocks = mf.part != nullptr ? mf.E : 0;
  DM_ARG_CHECK(T >= 0 && k >= 1 && k <= DECOMOE_MAX_TOPK, "dispatch: bad T=%lld or k=%d", (long long)T, k);
  DM_ARG_CHECK(K >= 1 && K <= DECOMOE_MAX_E, "dispatch: K=%d outside [1, %d]", K, DECOMOE_MAX_E);
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "dispatch: bad dtype");
  DM_ARG_CHECK(counts && offsets, "dispatch: counts/offsets null");
  const int64_t N = T * k;
  DM_ARG_CHECK(N < 0x7fffffffLL, "dispatch: T*k too large");
  DM_ARG_CHECK(N > 0 || mblocks == 0, "dispatch: a deferred mass needs routed pairs");
  if (N == 0) {
    DM_CUDA_CHECK(cudaMemsetAsync(counts, 0, sizeof(int32_t) * K, s));
    DM_CUDA_CHECK(cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (K + 1), s));
    return DECOMOE_OK;
  }
  DM_ARG_CHECK(topk_idx && perm_token && inv_slot, "dispatch: null index array");
  const size_t row_bytes = static_cast<size_t>(d) * dtype_bytes(dtype);
  if (x_perm != nullptr) {
    DM_ARG_CHECK(x != nullptr && d > 0, "dispatch: x null or d <= 0");
    DM_ARG_CHECK(row_bytes % 16 == 0 && aligned16(x) && aligned16(x_perm),
                 "dispatch: rows must be 16-byte multiples and 16-byte aligned");
  }
  if (ws == nullptr || ws_bytes < decomoe_dispatch_workspace_bytes(T, k, K)) {
    set_error("dispatch: workspace needs %zu bytes", decomoe_dispatch_workspace_bytes(T, k, K));
    return DECOMOE_ERR_WORKSPACE;
  }
  const int ntiles = static_cast<int>((N + DSP_TILE - 1) / DSP_TILE);
  int32_t* tile_hist = static_cast<int32_t*>(ws);
  if (ntiles == 1) {
    // one tile (decode sizes): count, scan and rank in one block, and copy
    // the rows there too when they are few
    const bool gather_here = x_perm != nullptr && static_cast<size_t>(N) * row_bytes <= 64 * 1024;
    DM_CUDA_CHECK(launch_pdl(k_dispatch_scatter<true>, dim3(1 + mblocks), dim3(DSP_THREADS), 0, s, topk_idx, N,
                             k, K, static_cast<const int32_t*>(nullptr), 1, counts, offsets, perm_token, inv_slot,
                             status_dev, static_cast<const uint4*>(x), static_cast<int>(row_bytes / 16),
                             gather_here ? static_cast<uint4*>(x_perm) : static_cast<uint4*>(nullptr), mf));
    if (gather_here) return DECOMOE_OK;
  } else {
    DM_CUDA_CHECK(launch_pdl(k_dispatch_hist, dim3(ntiles + mblocks), dim3(DSP_THREADS), 0, s, topk_idx, N, K,
                             tile_hist, status_dev, ntiles, mf));
    DM_CUDA_CHECK(launch_pdl(k_dispatch_scatter<false>, dim3(ntiles), dim3(DSP_THREADS), 0, s, topk_idx, N, k, K,
                             static_cast<const int32_t*>(tile_hist), ntiles, counts, offsets, perm_token, inv_slot,
                             static_cast<int32_t*>(nullptr), static_cast<const uint4*>(nullptr), 0,
                             static_cast<uint4*>(nullptr), MassFinish{}));
  }
  if (x_perm != nullptr) DM_RET(launch_gather_rows(x, perm_token, offsets, K, row_bytes, N, x_perm, s));
  return DECOMOE_OK;
}

int launch_gather_rows(const void* x, const int32_t* perm_token, const int32_t* offsets, int K, size_t row_bytes,
                       int64_t N, void* x_perm, cudaStream_t s) {
  const int vec = static_cast<int>(row_bytes / 16);
  int blocks = static_cast<int>(std::min<int64_t>((N * 32 + 255) / 256, sm_count() * 8LL));
  if (blocks < 1) blocks = 1;
  DM_CUDA_CHECK(launch_pdl(k_gather_rows, dim3(blocks), dim3(256), 0, s, static_cast<const uint4*>(x), perm_token,
                           offsets, K, vec, static_cast<uint4*>(x_perm)));
  return DECOMOE_OK;
}

}  // namespace decomoe

// ---------------------------------------------------------------------------
// Allocation-free dispatch.
//
// Some callers cannot hand the library a workspace: their runtime owns every
// device allocation up front (a serving engine that carves all of HBM into a
// fixed arena at start-up and forbids any later cudaMalloc, because cudaMalloc
// can synchronise the device and fragment that arena). For them this entry
// point keeps the per-tile histograms in a fixed array that is part of the
// library image itself, so the call needs nothing beyond its inputs and
// outputs.
//
// Limit: ceil(T*k / 1024) * K <= DECOMOE_NOALLOC_DISPATCH_SCRATCH_INTS
// (65536 int32 = 256 KiB, e.g. T*k up to 524288 pairs at K = 128). Every GPU
// that loads the library holds this array until the process exits.
// ---------------------------------------------------------------------------
namespace decomoe {

static __device__ __align__(256) int32_t g_noalloc_dispatch_scratch[DECOMOE_NOALLOC_DISPATCH_SCRATCH_INTS];

// Device address of the array, looked up once per device ordinal (host code
// cannot use the symbol itself as a device pointer). The cached address
// belongs to the device's primary context as it was at the first call: it is
// not looked up again after cudaDeviceReset. The first call on a device must
// not be made while `s` is being captured into a graph.
static int noalloc_scratch_ptr(int32_t** out, cudaStream_t s) {
  static std::mutex mu;
  static int32_t* ptrs[64] = {nullptr};
  int dev = 0;
  DM_CUDA_CHECK(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) {
    set_error("dispatch_noalloc: device ordinal %d out of range", dev);
    return DECOMOE_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lk(mu);
  if (ptrs[dev] == nullptr) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    DM_CUDA_CHECK(cudaStreamIsCapturing(s, &cs));
    if (cs != cudaStreamCaptureStatusNone) {
      set_error("dispatch_noalloc: the first call on device %d is inside a stream capture; make one call on "
                "this device before capturing", dev);
      return DECOMOE_ERR_INVALID_ARG;
    }
    void* p = nullptr;
    DM_CUDA_CHECK(cudaGetSymbolAddress(&p, g_noalloc_dispatch_scratch));
    ptrs[dev] = static_cast<int32_t*>(p);
  }
  *out = ptrs[dev];
  return DECOMOE_OK;
}

}  // namespace decomoe

extern "C" int decomoe_dispatch_noalloc(const int32_t* topk_idx, int64_t T, int k, int K, const void* x, int d,
                                        int dtype, int32_t* counts, int32_t* offsets, int32_t* perm_token,
                                        int32_t* inv_slot, void* x_perm, int32_t* status_dev,
                                        decomoe_stream_t stream) {
  using namespace decomoe;
  clear_error();
  DM_ARG_CHECK(T >= 0 && k >= 1 && k <= DECOMOE_MAX_TOPK, "dispatch_noalloc: bad T=%lld or k=%d", (long long)T, k);
  DM_ARG_CHECK(K >= 1 && K <= DECOMOE_MAX_E, "dispatch_noalloc: K=%d outside [1, %d]", K, DECOMOE_MAX_E);
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "dispatch_noalloc: bad dtype");
  DM_ARG_CHECK(counts && offsets, "dispatch_noalloc: counts/offsets null");
  const int64_t N = T * k;
  DM_ARG_CHECK(N < 0x7fffffffLL, "dispatch_noalloc: T*k too large");
  const int64_t ntiles64 = (N + DSP_TILE - 1) / DSP_TILE;
  DM_ARG_CHECK(ntiles64 * K <= DECOMOE_NOALLOC_DISPATCH_SCRATCH_INTS,
               "dispatch_noalloc: ceil(T*k/%d)*K = %lld exceeds the fixed scratch of %d entries; "
               "use decomoe_dispatch with a workspace", DSP_TILE, (long long)(ntiles64 * K),
               DECOMOE_NOALLOC_DISPATCH_SCRATCH_INTS);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (N == 0) {
    DM_CUDA_CHECK(cudaMemsetAsync(counts, 0, sizeof(int32_t) * K, s));
    DM_CUDA_CHECK(cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (K + 1), s));
    return DECOMOE_OK;
  }
  DM_ARG_CHECK(topk_idx && perm_token && inv_slot, "dispatch_noalloc: null index array");
  const size_t row_bytes = static_cast<size_t>(d) * dtype_bytes(dtype);
  if (x_perm != nullptr) {
    DM_ARG_CHECK(x != nullptr && d > 0, "dispatch_noalloc: x null or d <= 0");
    DM_ARG_CHECK(row_bytes % 16 == 0 && aligned16(x) && aligned16(x_perm),
                 "dispatch_noalloc: rows must be 16-byte multiples and 16-byte aligned");
  }
  int32_t* tile_hist = nullptr;
  DM_RET(noalloc_scratch_ptr(&tile_hist, s));
  // k_dispatch_hist writes every entry the scatter pass reads, so nothing
  // left in the array by an earlier call is ever used.
  const int ntiles = static_cast<int>(ntiles64);
  DM_CUDA_CHECK(launch_pdl(k_dispatch_hist, dim3(ntiles), dim3(DSP_THREADS), 0, s, topk_idx, N, K, tile_hist,
                           status_dev, ntiles, MassFinish{}));
  k_dispatch_scatter<false><<<ntiles, DSP_THREADS, 0, s>>>(topk_idx, N, k, K, tile_hist, ntiles, counts, offsets,
                                                    perm_token, inv_slot);
  DM_LAUNCH_CHECK("k_dispatch_scatter");
  if (x_perm != nullptr) DM_RET(launch_gather_rows(x, perm_token, offsets, K, row_bytes, N, x_perm, s));
  return DECOMOE_OK;
}
