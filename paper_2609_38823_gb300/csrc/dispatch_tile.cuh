// One dispatch tile (DecoMoE Algorithm 2: the routed (token, slot) pairs
// grouped by prefix expert): the stable count, scan and rank of
// DSP_TILE = 1024 consecutive pairs by one block of 256 threads, shared by
// the dispatch kernels and by the single routing block of the decode sizes,
// which dispatches its own picks without a further launch.
#pragma once

#include "decomoe_internal.cuh"

namespace decomoe {

constexpr int DSP_THREADS = 256;
constexpr int DSP_WARPS = DSP_THREADS / 32;
constexpr int DSP_PER_WARP = 128;                   // consecutive pairs per warp
constexpr int DSP_TILE = DSP_WARPS * DSP_PER_WARP;  // pairs per block (1024)

// Pass 2: every block sums the tile histograms (its own prefix and the total),
// scans the totals over experts, then ranks its pairs stably: warp w owns
// pairs [w*128, w*128+128) of the tile in order, ranks inside a 32-pair round
// come from __match_any_sync, and per-warp running counts are scanned across
// warps. Writes perm_token and inv_slot; block 0 writes counts and offsets.
// SINGLE: one tile in one block (decode sizes): the block also counts the
// histogram itself and may copy the rows (x_perm != null); blocks from 1 on
// finish a deferred mass.
// Called by all DSP_THREADS threads of the block; tile = this block's tile
// index (0 with SINGLE).
template <bool SINGLE>
__device__ __forceinline__ void dispatch_tile(const int32_t* __restrict__ idx, int64_t N, int k, int K,
                                              const int32_t* __restrict__ tile_hist, int ntiles, int tile,
                                              int32_t* __restrict__ counts, int32_t* __restrict__ offsets,
                                              int32_t* __restrict__ perm_token, int32_t* __restrict__ inv_slot,
                                              int32_t* status, const uint4* __restrict__ x, int row_vec,
                                              uint4* __restrict__ x_perm) {
  __shared__ int s_base[DECOMOE_MAX_E];
  __shared__ int s_wcnt[DSP_WARPS][DECOMOE_MAX_E];
  __shared__ int s_wsum[DSP_WARPS];
  __shared__ int s_row[SINGLE ? DSP_TILE : 1];  // rows of this tile's pairs (for the in-block gather)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int e_t = threadIdx.x;  // one expert per thread (K <= 256 = DSP_THREADS)

  int tot = 0, before = 0;
  if constexpr (SINGLE) {
    // a single tile (one block): count its pairs here, as k_dispatch_hist does
    int* s_cnt = &s_wcnt[0][0];
    for (int e = threadIdx.x; e < K; e += DSP_THREADS) s_cnt[e] = 0;
    __syncthreads();
#pragma unroll
    for (int r = 0; r < DSP_PER_WARP / 32; ++r) {
      const int64_t f = static_cast<int64_t>(warp) * DSP_PER_WARP + r * 32 + lane;
      int e = -2;
      if (f < N) {
        e = idx[f];
        if (e < 0 || e >= K) {
          report_status(status, DECOMOE_ERR_BAD_INPUT);
          e = -1;
        }
      }
      const uint32_t grp = __match_any_sync(0xffffffffu, e);
      if (e >= 0 && lane == __ffs(grp) - 1) atomicAdd(&s_cnt[e], __popc(grp));
    }
    __syncthreads();
    if (e_t < K) tot = s_cnt[e_t];
    __syncthreads();
  } else if (e_t < K) {
    for (int b = 0; b < ntiles; ++b) {
      const int v = tile_hist[static_cast<int64_t>(b) * K + e_t];
      tot += v;
      if (b < tile) before += v;
    }
  }
  // exclusive block scan of tot over experts
  int incl = tot;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += v;
  }
  if (lane == 31) s_wsum[warp] = incl;
  for (int e = threadIdx.x; e < K; e += DSP_THREADS)
    for (int w = 0; w < DSP_WARPS; ++w) s_wcnt[w][e] = 0;
  __syncthreads();
  int wpre = 0;
  for (int w = 0; w < warp; ++w) wpre += s_wsum[w];
  const int excl = wpre + incl - tot;
  if (e_t < K) {
    s_base[e_t] = excl + before;
    if (tile == 0) {
      counts[e_t] = tot;
      offsets[e_t] = excl;
      if (e_t == K - 1) offsets[K] = excl + tot;
    }
  }
  __syncthreads();

  const int64_t base = static_cast<int64_t>(tile) * DSP_TILE + warp * DSP_PER_WARP;
  int rank[DSP_PER_WARP / 32];
  int ex[DSP_PER_WARP / 32];
#pragma unroll
  for (int r = 0; r < DSP_PER_WARP / 32; ++r) {
    const int64_t f = base + r * 32 + lane;
    int e = -2;
    if (f < N) {
      e = idx[f];
      if (e < 0 || e >= K) e = -1;
    }
    const uint32_t grp = __match_any_sync(0xffffffffu, e);
    const uint32_t lt = (1u << lane) - 1u;
    int rk = 0;
    if (e >= 0) rk = s_wcnt[warp][e] + __popc(grp & lt);
    __syncwarp();
    if (e >= 0 && lane == __ffs(grp) - 1) s_wcnt[warp][e] += __popc(grp);
    __syncwarp();
    rank[r] = rk;
    ex[r] = e;
  }
  __syncthreads();
  // per-expert exclusive scan over warps
  for (int e = threadIdx.x; e < K; e += DSP_THREADS) {
    int run = 0;
    for (int w = 0; w < DSP_WARPS; ++w) {
      const int c = s_wcnt[w][e];
      s_wcnt[w][e] = run;
      run += c;
    }
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < DSP_PER_WARP / 32; ++r) {
    const int64_t f = base + r * 32 + lane;
    if (f >= N) continue;
    const int e = ex[r];
    int row = -1;
    if (e >= 0) {
      row = s_base[e] + s_wcnt[warp][e] + rank[r];
      perm_token[row] = static_cast<int32_t>(f / k);
    }
    inv_slot[f] = row;
    if constexpr (SINGLE) s_row[warp * DSP_PER_WARP + r * 32 + lane] = row;
  }
  if (!SINGLE || x_perm == nullptr) return;
  // in-block gather (single small tile): warp per pair, 16-byte vectors
  __syncthreads();
  const int64_t n_here = (N - static_cast<int64_t>(tile) * DSP_TILE < DSP_TILE)
                             ? N - static_cast<int64_t>(tile) * DSP_TILE
                             : DSP_TILE;
  for (int i = warp; i < n_here; i += DSP_WARPS) {
    const int row = s_row[i];
    if (row < 0) continue;
    const int64_t f = static_cast<int64_t>(tile) * DSP_TILE + i;
    const uint4* src = x + (f / k) * row_vec;
    uint4* dst = x_perm + static_cast<int64_t>(row) * row_vec;
    int c = lane;
    for (; c + 32 * 3 < row_vec; c += 32 * 4) {
      uint4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = __ldg(src + c + 32 * u);
#pragma unroll
      for (int u = 0; u < 4; ++u) dst[c + 32 * u] = v[u];
    }
    for (; c < row_vec; c += 32) dst[c] = __ldg(src + c);
  }
}

}  // namespace decomoe
