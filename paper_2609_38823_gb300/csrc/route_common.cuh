// Device helpers of the routing step (DecoMoE Section 3.3, Eqs. 10-12)
// shared by the routing kernels and the one-launch decode layer: the
// order-preserving float keys and warp arg-max top-k, the renormalised pick
// weights, Eq. 12 on the device, and the bf16 dot product of the router's
// CUDA-core path.
#pragma once

#include "decomoe_internal.cuh"

namespace decomoe {

constexpr int GEMV_THREADS = 128;
constexpr int GEMV_TPB = 8;  // tokens per block
constexpr int GEMV_VPT = 2;  // vectors per thread per pass (d = 2048: one pass)
__device__ __forceinline__ float dot8_bf16(const uint4 a, const uint4 b, float acc) {
  acc = fmaf(bf16_lo(a.x), bf16_lo(b.x), acc);
  acc = fmaf(bf16_hi(a.x), bf16_hi(b.x), acc);
  acc = fmaf(bf16_lo(a.y), bf16_lo(b.y), acc);
  acc = fmaf(bf16_hi(a.y), bf16_hi(b.y), acc);
  acc = fmaf(bf16_lo(a.z), bf16_lo(b.z), acc);
  acc = fmaf(bf16_hi(a.z), bf16_hi(b.z), acc);
  acc = fmaf(bf16_lo(a.w), bf16_lo(b.w), acc);
  acc = fmaf(bf16_hi(a.w), bf16_hi(b.w), acc);
  return acc;
}

// Order-preserving 32-bit key of a float (larger float -> larger key; -0 and
// +0 share a key so equal values tie). Key 0 is below every float's key and
// marks entries that are out of range or already picked.
__device__ __forceinline__ uint32_t fkey(float f) {
  const uint32_t u = (f == 0.0f) ? 0u : __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float fkey_inv(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// k rounds of warp arg-max over entries e < lim (entry lane + 32 i in slot
// i; NSL slots cover 32 NSL entries): each round one redux.sync max over the
// lanes' best keys; when a single lane holds that key (no tie) a ballot
// names it, otherwise one redux.sync min over the indices of the lanes
// holding it picks the lower index. Only the winning lane clears its key, so
// the next round waits on nothing else; pick j ends in lane j.
template <int NSL>
__device__ __forceinline__ void warp_topk_n(const uint32_t (&key_in)[NSL], int lim, int k, int lane, float& my_v,
                                            int& my_i) {
  uint32_t key[NSL];
#pragma unroll
  for (int i = 0; i < NSL; ++i) key[i] = (lane + 32 * i < lim) ? key_in[i] : 0u;
  my_v = 0.f;
  my_i = 0;
  for (int j = 0; j < k; ++j) {
    uint32_t bk = 0;
    int bs = 0;  // slot of the lane's best (entries ascend with the slot, so strict > keeps the lowest index)
#pragma unroll
    for (int i = 0; i < NSL; ++i)
      if (key[i] > bk) {
        bk = key[i];
        bs = i;
      }
    const uint32_t mk = __reduce_max_sync(0xffffffffu, bk);
    const uint32_t bal = __ballot_sync(0xffffffffu, bk == mk);
    int wl, ws;  // winning lane and its slot (ws valid in lane wl)
    if ((bal & (bal - 1u)) == 0u) {
      wl = __ffs(bal) - 1;
      ws = bs;
    } else {
      const uint32_t cand = (bk == mk) ? static_cast<uint32_t>(lane + 32 * bs) : 0xffffffffu;
      const uint32_t wi = __reduce_min_sync(0xffffffffu, cand);
      wl = static_cast<int>(wi & 31u);
      ws = static_cast<int>(wi >> 5);
    }
    {
      const bool mine = wl == lane;
#pragma unroll
      for (int i = 0; i < NSL; ++i) key[i] = (mine && i == ws) ? 0u : key[i];  // selects keep key[] in registers
    }
    const int wi = wl + 32 * __shfl_sync(0xffffffffu, ws, wl);
    if (lane == j) {
      my_v = fkey_inv(mk);
      my_i = wi;
    }
  }
}

__device__ __forceinline__ void warp_topk(const uint32_t (&key_in)[8], int lim, int k, int lane, float& my_v,
                                          int& my_i) {
  warp_topk_n<8>(key_in, lim, k, lane, my_v, my_i);
}

// Renormalised weight of this lane's pick (lanes >= k get 0).
__device__ __forceinline__ float pick_weight(float my_v, int lane, int k) {
  const float v0 = __shfl_sync(0xffffffffu, my_v, 0);
  const float z = (lane < k) ? __expf(my_v - v0) : 0.f;
  float zs = z;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) zs += __shfl_xor_sync(0xffffffffu, zs, off);
  return z / zs;
}

// Eq. 12, sequentially in fp64 with round-to-nearest adds and division, as
// the host decomoe_select_prefix does: K_hat = smallest K whose prefix mass
// ratio reaches p (E when p >= 1 or none does), K = max(k, K_hat); k when the
// total mass is zero.
__device__ __forceinline__ int select_prefix_seq(const double* mass, int E, int k, double p) {
  double tot = 0.0;
  for (int e = 0; e < E; ++e) tot = __dadd_rn(tot, mass[e]);
  int K = k;
  if (tot > 0.0) {
    int K_hat = E;
    if (p < 1.0) {
      double acc = 0.0;
      for (int Kc = 1; Kc <= E; ++Kc) {
        acc = __dadd_rn(acc, mass[Kc - 1]);
        if (__ddiv_rn(acc, tot) >= p) {
          K_hat = Kc;
          break;
        }
      }
    }
    K = K_hat > k ? K_hat : k;
  }
  return K;
}

}  // namespace decomoe
