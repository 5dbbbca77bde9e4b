// Combine of the expert outputs (DecoMoE Algorithm 2: "evaluate and combine"),
// visual-block removal from hidden states and KV rows (Section 3.2), and the
// RMSNorm of the attention-free layer stack. All three are HBM-bound copies
// or reductions over rows: 16-byte vector accesses, one warp per row.
#include "decomoe_internal.cuh"

namespace decomoe {

// ------------------------------------------------------------------ combine
// out[t] = sum_j w[t, j] * y[inv_slot[t*k + j]] (+ residual[t]); one warp per
// token, lane handles 8 bf16 (or 4 fp32) columns per 16-byte vector. For
// k <= 8 the slot rows and weights sit in registers and the k row loads of a
// vector position are issued together before the fp32 sum in slot order
// j = 0..k-1; larger k takes a loop with the same order.
template <bool BF16>
__device__ __forceinline__ void acc_vec(float* acc, const uint4& v, float wj) {
  if constexpr (BF16) {
    acc[0] = fmaf(wj, bf16_lo(v.x), acc[0]);
    acc[1] = fmaf(wj, bf16_hi(v.x), acc[1]);
    acc[2] = fmaf(wj, bf16_lo(v.y), acc[2]);
    acc[3] = fmaf(wj, bf16_hi(v.y), acc[3]);
    acc[4] = fmaf(wj, bf16_lo(v.z), acc[4]);
    acc[5] = fmaf(wj, bf16_hi(v.z), acc[5]);
    acc[6] = fmaf(wj, bf16_lo(v.w), acc[6]);
    acc[7] = fmaf(wj, bf16_hi(v.w), acc[7]);
  } else {
    acc[0] = fmaf(wj, __uint_as_float(v.x), acc[0]);
    acc[1] = fmaf(wj, __uint_as_float(v.y), acc[1]);
    acc[2] = fmaf(wj, __uint_as_float(v.z), acc[2]);
    acc[3] = fmaf(wj, __uint_as_float(v.w), acc[3]);
  }
}

template <bool BF16>
__device__ __forceinline__ uint4 finish_vec(float* acc, const uint4* __restrict__ residual, int64_t ridx) {
  if (residual != nullptr) acc_vec<BF16>(acc, __ldg(residual + ridx), 1.0f);
  if constexpr (BF16)
    return make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                      pack_bf16x2(acc[6], acc[7]));
  else
    return make_uint4(__float_as_uint(acc[0]), __float_as_uint(acc[1]), __float_as_uint(acc[2]),
                      __float_as_uint(acc[3]));
}

// Visual-block removal fused into the combine: every output vector of a text
// row (t < v0 or t >= v0 + nv) is also stored to text[t'] with t' = t, or
// t - nv past the block: the rows decomoe_drop_visual_block would copy from
// out, written while they are in registers.
struct DropRows {
  uint4* text = nullptr;  // null: no second store
  int64_t v0 = 0, nv = 0;
};

// WPT warps per token, each taking alternate 32-vector chunks of the row:
// many tokens take one warp each (two blocks resident per SM), few tokens
// spread each row over more warps.
// discard (y is the caller's scratch, rows 128-byte aligned): every y line is
// read exactly once (inv_slot is a bijection), so once a warp has summed its
// rows it drops their L2 lines (discard.global.L2): the lines are not written
// back to HBM, and the next writer of the scratch finds clean lines to evict.
__device__ __forceinline__ void l2_discard_line(const void* p) {
  asm volatile("discard.global.L2 [%0], 128;" ::"l"(p) : "memory");
}

template <bool BF16, int KT, bool DROP, int WPT>
__global__ void __launch_bounds__(256, WPT == 1 ? 2 : 1)
    k_combine(const uint4* __restrict__ y, const int32_t* __restrict__ inv_slot,
              const float* __restrict__ w, int64_t Tn, int k, int vec,
              const uint4* __restrict__ residual, uint4* __restrict__ out, DropRows drop, int discard) {
  pdl_enter();
  constexpr int NE = BF16 ? 8 : 4;
  const int lane = threadIdx.x & 31;
  const int64_t gw = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t wt = gw; wt < Tn * WPT; wt += nw) {
    const int64_t t = wt / WPT;
    const int part = static_cast<int>(wt - t * WPT);
    const bool text_row = DROP && (t < drop.v0 || t >= drop.v0 + drop.nv);
    const int64_t trow = t < drop.v0 ? t : t - drop.nv;
    int my_row = -1;
    float my_w = 0.f;
    if (lane < k) {
      my_row = inv_slot[t * k + lane];
      my_w = w[t * k + lane];
    }
    if constexpr (KT > 0) {
      int rows[KT];
      float wts[KT];
#pragma unroll
      for (int j = 0; j < KT; ++j) {
        rows[j] = __shfl_sync(0xffffffffu, my_row, j);
        wts[j] = __shfl_sync(0xffffffffu, my_w, j);
      }
      // two chunks (64 vectors apart) per iteration: 2*KT loads in flight
      for (int c = part * 32 + lane; c < vec; c += 64 * WPT) {
        const int c2 = c + 32 * WPT;
        const bool two = c2 < vec;
        uint4 v[KT], v2[KT];
#pragma unroll
        for (int j = 0; j < KT; ++j) {
          v[j] = rows[j] >= 0 ? __ldg(y + static_cast<int64_t>(rows[j]) * vec + c) : make_uint4(0, 0, 0, 0);
          v2[j] = (rows[j] >= 0 && two) ? __ldg(y + static_cast<int64_t>(rows[j]) * vec + c2) : make_uint4(0, 0, 0, 0);
        }
        float acc[NE], acc2[NE];
#pragma unroll
        for (int i = 0; i < NE; ++i) acc[i] = acc2[i] = 0.f;
#pragma unroll
        for (int j = 0; j < KT; ++j)
          if (rows[j] >= 0) {
            acc_vec<BF16>(acc, v[j], wts[j]);
            acc_vec<BF16>(acc2, v2[j], wts[j]);
          }
        if (discard) {
          // every lane's loads of these lines have been consumed above
          __syncwarp();
          if ((lane & 7) == 0) {
#pragma unroll
            for (int j = 0; j < KT; ++j)
              if (rows[j] >= 0) {
                l2_discard_line(y + static_cast<int64_t>(rows[j]) * vec + c);
                if (two) l2_discard_line(y + static_cast<int64_t>(rows[j]) * vec + c2);
              }
          }
        }
        const uint4 o1 = finish_vec<BF16>(acc, residual, t * vec + c);
        out[t * vec + c] = o1;
        if (text_row) drop.text[trow * vec + c] = o1;
        if (two) {
          const uint4 o2 = finish_vec<BF16>(acc2, residual, t * vec + c2);
          out[t * vec + c2] = o2;
          if (text_row) drop.text[trow * vec + c2] = o2;
        }
      }
    } else {
      for (int c0 = part * 32; c0 < vec; c0 += 32 * WPT) {
        // every lane takes part in the shuffles; only lanes with c < vec load/store
        const int c = c0 + lane;
        const bool active = c < vec;
        float acc[NE];
#pragma unroll
        for (int i = 0; i < NE; ++i) acc[i] = 0.f;
        for (int j = 0; j < k; ++j) {
          const int row = __shfl_sync(0xffffffffu, my_row, j);
          const float wj = __shfl_sync(0xffffffffu, my_w, j);
          if (row < 0 || !active) continue;
          acc_vec<BF16>(acc, __ldg(y + static_cast<int64_t>(row) * vec + c), wj);
        }
        if (active) {
          const uint4 o1 = finish_vec<BF16>(acc, residual, t * vec + c);
          out[t * vec + c] = o1;
          if (text_row) drop.text[trow * vec + c] = o1;
        }
      }
    }
  }
}

static int grid_for_warps(int64_t warps);

template <bool BF16, bool DROP, int WPT>
static cudaError_t launch_combine_w(cudaStream_t s, const uint4* y, const int32_t* inv, const float* w, int64_t T,
                                    int k, int vec, const uint4* res, uint4* out, DropRows drop, int dc) {
  const dim3 g(grid_for_warps(WPT * T)), b(256);
  switch (k) {
    case 1: return launch_pdl(k_combine<BF16, 1, DROP, WPT>, g, b, 0, s, y, inv, w, T, k, vec, res, out, drop, dc);
    case 2: return launch_pdl(k_combine<BF16, 2, DROP, WPT>, g, b, 0, s, y, inv, w, T, k, vec, res, out, drop, dc);
    case 4: return launch_pdl(k_combine<BF16, 4, DROP, WPT>, g, b, 0, s, y, inv, w, T, k, vec, res, out, drop, dc);
    case 8: return launch_pdl(k_combine<BF16, 8, DROP, WPT>, g, b, 0, s, y, inv, w, T, k, vec, res, out, drop, dc);
    default: return launch_pdl(k_combine<BF16, 0, DROP, WPT>, g, b, 0, s, y, inv, w, T, k, vec, res, out, drop, 0);
  }
}
// Warps per token by token count: one from 1024 tokens on, two from 256, four
// from 32, eight below (a decode step's row then spans eight warps).
template <bool BF16, bool DROP>
static cudaError_t launch_combine_k(cudaStream_t s, const uint4* y, const int32_t* inv, const float* w, int64_t T,
                                    int k, int vec, const uint4* res, uint4* out, DropRows drop, int dc) {
  if (T >= 1024) return launch_combine_w<BF16, DROP, 1>(s, y, inv, w, T, k, vec, res, out, drop, dc);
  if (T >= 256) return launch_combine_w<BF16, DROP, 2>(s, y, inv, w, T, k, vec, res, out, drop, dc);
  if (T >= 32) return launch_combine_w<BF16, DROP, 4>(s, y, inv, w, T, k, vec, res, out, drop, dc);
  return launch_combine_w<BF16, DROP, 8>(s, y, inv, w, T, k, vec, res, out, drop, dc);
}
template <bool BF16>
static cudaError_t launch_combine(cudaStream_t s, const uint4* y, const int32_t* inv, const float* w, int64_t T,
                                  int k, int vec, const uint4* res, uint4* out, DropRows drop, int dc) {
  return drop.text != nullptr ? launch_combine_k<BF16, true>(s, y, inv, w, T, k, vec, res, out, drop, dc)
                              : launch_combine_k<BF16, false>(s, y, inv, w, T, k, vec, res, out, drop, dc);
}

// ------------------------------------------------------------------ compaction
// dst[b, r'] = src[b, r'] for r' < v0, src[b, r' + nv] otherwise. A flat grid
// over the output's 16-byte vectors (batch, row, column; column fastest, so a
// warp moves 512 contiguous bytes), four vectors per thread in flight.
// flag (optional): the removal runs only when *flag == 1 (the SAVB gate's
// exit decision, read on the device); any other value leaves dst untouched.
__global__ void __launch_bounds__(256)
    k_compact_vec(const uint4* __restrict__ src, uint4* __restrict__ dst, int64_t rows_out,
                  int64_t vec, int64_t v0, int64_t nv, int64_t nbatch, int64_t sstride,
                  int64_t dstride, const int32_t* __restrict__ flag) {
  pdl_enter();
  if (flag != nullptr && *flag != 1) return;
  constexpr int U = 4;
  const int64_t total = nbatch * rows_out * vec;
  const int64_t step = static_cast<int64_t>(gridDim.x) * blockDim.x * U;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x * U + threadIdx.x; base < total; base += step) {
    uint4 v[U];
    int64_t di[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t i = base + static_cast<int64_t>(u) * blockDim.x;
      di[u] = -1;
      if (i < total) {
        const int64_t c = i % vec;
        const int64_t q = i / vec;
        const int64_t b = q / rows_out;
        const int64_t r = q - b * rows_out;
        const int64_t rs = r < v0 ? r : r + nv;
        v[u] = __ldcs(src + b * sstride + rs * vec + c);
        di[u] = b * dstride + r * vec + c;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (di[u] >= 0) __stcs(dst + di[u], v[u]);
  }
}

// Byte path for rows or strides that are not 16-byte multiples.
__global__ void k_compact_bytes(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                int64_t rows_out, int64_t row_bytes, int64_t v0, int64_t nv,
                                int64_t nbatch, int64_t sstride, int64_t dstride, const int32_t* __restrict__ flag) {
  pdl_enter();
  if (flag != nullptr && *flag != 1) return;
  const int64_t total = nbatch * rows_out * row_bytes;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t c = i % row_bytes;
    const int64_t q = i / row_bytes;
    const int64_t b = q / rows_out;
    const int64_t r = q - b * rows_out;
    const int64_t rs = r < v0 ? r : r + nv;
    dst[b * dstride + r * row_bytes + c] = src[b * sstride + rs * row_bytes + c];
  }
}

// ------------------------------------------------------------------ RMSNorm
template <bool BF16>
__global__ void __launch_bounds__(256)
    k_rmsnorm(const uint4* __restrict__ x, uint4* __restrict__ y, int64_t Tn, int vec, int d,
              float eps) {
  pdl_enter();
  const int lane = threadIdx.x & 31;
  const int64_t gw = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t t = gw; t < Tn; t += nw) {
    const uint4* xr = x + t * vec;
    float ss = 0.f;
    for (int c = lane; c < vec; c += 32) {
      const uint4 v = xr[c];
      if constexpr (BF16) {
        const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float a = bf16_lo(u[i]), b = bf16_hi(u[i]);
          ss = fmaf(a, a, ss);
          ss = fmaf(b, b, ss);
        }
      } else {
        const float a[4] = {__uint_as_float(v.x), __uint_as_float(v.y), __uint_as_float(v.z),
                            __uint_as_float(v.w)};
#pragma unroll
        for (int i = 0; i < 4; ++i) ss = fmaf(a[i], a[i], ss);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    const float inv = rsqrtf(ss / static_cast<float>(d) + eps);
    uint4* yr = y + t * vec;
    for (int c = lane; c < vec; c += 32) {
      const uint4 v = xr[c];
      uint4 o;
      if constexpr (BF16) {
        o.x = pack_bf16x2(bf16_lo(v.x) * inv, bf16_hi(v.x) * inv);
        o.y = pack_bf16x2(bf16_lo(v.y) * inv, bf16_hi(v.y) * inv);
        o.z = pack_bf16x2(bf16_lo(v.z) * inv, bf16_hi(v.z) * inv);
        o.w = pack_bf16x2(bf16_lo(v.w) * inv, bf16_hi(v.w) * inv);
      } else {
        o.x = __float_as_uint(__uint_as_float(v.x) * inv);
        o.y = __float_as_uint(__uint_as_float(v.y) * inv);
        o.z = __float_as_uint(__uint_as_float(v.z) * inv);
        o.w = __float_as_uint(__uint_as_float(v.w) * inv);
      }
      yr[c] = o;
    }
  }
}

static int grid_for_warps(int64_t warps) {
  const int64_t want = (warps * 32 + 255) / 256;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  return static_cast<int>(std::max<int64_t>(1, std::min(want, cap)));
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

int decomoe_combine(const void* y_perm, const int32_t* inv_slot, const float* topk_w, int64_t T, int k,
                    int d, int dtype, const void* residual, void* out, decomoe_stream_t stream) {
  clear_error();
  return combine_impl(y_perm, inv_slot, topk_w, T, k, d, dtype, residual, out, nullptr, 0, 0, stream);
}

int decomoe_combine_drop_visual_block(const void* y_perm, const int32_t* inv_slot, const float* topk_w, int64_t T,
                                      int k, int d, int dtype, const void* residual, void* out, void* text_out,
                                      int64_t v0, int64_t nv, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(v0 >= 0 && nv >= 0 && v0 + nv <= T,
               "combine_drop_visual_block: visual block [%lld, %lld) outside [0, %lld)", (long long)v0,
               (long long)(v0 + nv), (long long)T);
  const bool any_text = T - nv > 0;  // an all-visual sequence leaves no text row to store
  DM_ARG_CHECK(text_out != nullptr || !any_text, "combine_drop_visual_block: text_out is null");
  return combine_impl(y_perm, inv_slot, topk_w, T, k, d, dtype, residual, out, any_text ? text_out : nullptr, v0,
                      nv, stream);
}

}  // extern "C"

namespace decomoe {

int combine_impl(const void* y_perm, const int32_t* inv_slot, const float* topk_w, int64_t T, int k, int d,
                 int dtype, const void* residual, void* out, void* text_out, int64_t v0, int64_t nv,
                 decomoe_stream_t stream, bool discard_y) {
  DM_ARG_CHECK(T >= 0 && k >= 1 && k <= DECOMOE_MAX_TOPK && d > 0, "combine: bad sizes");
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "combine: bad dtype");
  if (T == 0) return DECOMOE_OK;
  DM_ARG_CHECK(y_perm && inv_slot && topk_w && out, "combine: null pointer");
  const size_t row_bytes = static_cast<size_t>(d) * dtype_bytes(dtype);
  DM_ARG_CHECK(row_bytes % 16 == 0 && aligned16(y_perm) && aligned16(out) &&
                   (residual == nullptr || aligned16(residual)),
               "combine: rows must be 16-byte multiples, pointers 16-byte aligned");
  DM_ARG_CHECK(out != y_perm, "combine: out aliases y_perm");
  DropRows drop;
  if (text_out != nullptr) {
    DM_ARG_CHECK(v0 >= 0 && nv >= 0 && v0 + nv <= T, "combine: visual block [%lld, %lld) outside [0, %lld)",
                 (long long)v0, (long long)(v0 + nv), (long long)T);
    DM_ARG_CHECK(aligned16(text_out), "combine: text_out must be 16-byte aligned");
    const uintptr_t o0 = reinterpret_cast<uintptr_t>(out), o1 = o0 + static_cast<uintptr_t>(T) * row_bytes;
    const uintptr_t t0 = reinterpret_cast<uintptr_t>(text_out), t1 = t0 + static_cast<uintptr_t>(T - nv) * row_bytes;
    DM_ARG_CHECK(o1 <= t0 || t1 <= o0, "combine: text_out overlaps out");
    drop.text = static_cast<uint4*>(text_out);
    drop.v0 = v0;
    drop.nv = nv;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int vec = static_cast<int>(row_bytes / 16);
  // whole 128-byte lines only
  const int dc = discard_y && row_bytes % 128 == 0 && reinterpret_cast<uintptr_t>(y_perm) % 128 == 0 ? 1 : 0;
  if (dtype == DECOMOE_BF16)
    DM_CUDA_CHECK(launch_combine<true>(s, static_cast<const uint4*>(y_perm), inv_slot, topk_w, T, k, vec,
                                       static_cast<const uint4*>(residual), static_cast<uint4*>(out), drop, dc));
  else
    DM_CUDA_CHECK(launch_combine<false>(s, static_cast<const uint4*>(y_perm), inv_slot, topk_w, T, k, vec,
                                        static_cast<const uint4*>(residual), static_cast<uint4*>(out), drop, dc));
  return DECOMOE_OK;
}

}  // namespace decomoe

extern "C" {

int decomoe_drop_visual_block(const void* src, void* dst, int64_t rows, int64_t row_bytes, int64_t v0,
                              int64_t nv, int64_t nbatch, int64_t src_batch_stride,
                              int64_t dst_batch_stride, decomoe_stream_t stream) {
  clear_error();
  return drop_visual_block_impl(nullptr, src, dst, rows, row_bytes, v0, nv, nbatch, src_batch_stride,
                                dst_batch_stride, stream);
}

int decomoe_drop_visual_block_if(const int32_t* exit_flag, const void* src, void* dst, int64_t rows,
                                 int64_t row_bytes, int64_t v0, int64_t nv, int64_t nbatch,
                                 int64_t src_batch_stride, int64_t dst_batch_stride, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(exit_flag != nullptr, "drop_visual_block_if: exit_flag is null");
  return drop_visual_block_impl(exit_flag, src, dst, rows, row_bytes, v0, nv, nbatch, src_batch_stride,
                                dst_batch_stride, stream);
}

}  // extern "C"

namespace decomoe {

int drop_visual_block_impl(const int32_t* flag, const void* src, void* dst, int64_t rows, int64_t row_bytes,
                           int64_t v0, int64_t nv, int64_t nbatch, int64_t src_batch_stride,
                           int64_t dst_batch_stride, decomoe_stream_t stream) {
  DM_ARG_CHECK(rows >= 0 && row_bytes > 0 && nbatch >= 0, "drop_visual_block: bad sizes");
  DM_ARG_CHECK(v0 >= 0 && nv >= 0 && v0 + nv <= rows, "drop_visual_block: block [%lld, %lld) outside [0, %lld)",
               (long long)v0, (long long)(v0 + nv), (long long)rows);
  const int64_t rows_out = rows - nv;
  if (nbatch == 0 || rows_out == 0) return DECOMOE_OK;
  DM_ARG_CHECK(src && dst, "drop_visual_block: null pointer");
  DM_ARG_CHECK(nbatch == 1 || (src_batch_stride >= rows * row_bytes && dst_batch_stride >= rows_out * row_bytes),
               "drop_visual_block: batch strides smaller than a batch");
  {
    // src and dst ranges must not overlap
    const uintptr_t s0 = reinterpret_cast<uintptr_t>(src);
    const uintptr_t s1 = s0 + static_cast<uintptr_t>((nbatch - 1) * src_batch_stride + rows * row_bytes);
    const uintptr_t d0 = reinterpret_cast<uintptr_t>(dst);
    const uintptr_t d1 = d0 + static_cast<uintptr_t>((nbatch - 1) * dst_batch_stride + rows_out * row_bytes);
    DM_ARG_CHECK(s1 <= d0 || d1 <= s0, "drop_visual_block: src and dst overlap");
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const bool vec_ok = row_bytes % 16 == 0 && aligned16(src) && aligned16(dst) &&
                      (nbatch == 1 || (src_batch_stride % 16 == 0 && dst_batch_stride % 16 == 0));
  if (vec_ok) {
    const int64_t nvec = nbatch * rows_out * (row_bytes / 16);
    const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>((nvec + 1023) / 1024, sm_count() * 16LL)));
    DM_CUDA_CHECK(launch_pdl(k_compact_vec, dim3(grid), dim3(256), 0, s, static_cast<const uint4*>(src),
                             static_cast<uint4*>(dst), rows_out, row_bytes / 16, v0, nv, nbatch,
                             src_batch_stride / 16, dst_batch_stride / 16, flag));
  } else {
    const int grid = sm_count() * 8;
    DM_CUDA_CHECK(launch_pdl(k_compact_bytes, dim3(grid), dim3(256), 0, s, static_cast<const uint8_t*>(src),
                             static_cast<uint8_t*>(dst), rows_out, row_bytes, v0, nv, nbatch, src_batch_stride,
                             dst_batch_stride, flag));
  }
  return DECOMOE_OK;
}

}  // namespace decomoe

extern "C" {

int decomoe_rmsnorm(const void* x, void* y, int64_t T, int d, float eps, int dtype, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(T >= 0 && d > 0 && eps >= 0.f, "rmsnorm: bad sizes");
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "rmsnorm: bad dtype");
  if (T == 0) return DECOMOE_OK;
  DM_ARG_CHECK(x && y, "rmsnorm: null pointer");
  const size_t row_bytes = static_cast<size_t>(d) * dtype_bytes(dtype);
  DM_ARG_CHECK(row_bytes % 16 == 0 && aligned16(x) && aligned16(y), "rmsnorm: rows must be 16-byte multiples");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int vec = static_cast<int>(row_bytes / 16);
  const int grid = grid_for_warps(T);
  if (dtype == DECOMOE_BF16)
    DM_CUDA_CHECK(launch_pdl(k_rmsnorm<true>, dim3(grid), dim3(256), 0, s, static_cast<const uint4*>(x),
                             static_cast<uint4*>(y), T, vec, d, eps));
  else
    DM_CUDA_CHECK(launch_pdl(k_rmsnorm<false>, dim3(grid), dim3(256), 0, s, static_cast<const uint4*>(x),
                             static_cast<uint4*>(y), T, vec, d, eps));
  return DECOMOE_OK;
}

}  // extern "C"
