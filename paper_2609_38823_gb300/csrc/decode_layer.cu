// One launch per decode-size MoE layer (DecoMoE Algorithm 2: prefix-restricted
// routing repeated at every decoding step; Eqs. 10-12): router logits over the
// full pool, activated mass and device-side prefix, prefix top-k routing,
// dispatch, the grouped SwiGLU experts and the combine, for up to
// DL_MAX_T tokens, in a single persistent kernel.
//
// At decode sizes a layer step moves D x 9.4 MB of expert weights (D active
// experts) and almost nothing else, so its floor is the weight stream; with one
// launch per step the dependent launches of the separate calls (router,
// routing + dispatch, two expert GEMMs, combine) no longer sit between the
// step's start and the first weight byte, nor after the last one.
//
// Phases (one CTA per SM, every CTA resident):
//  A  router: CTA c computes logits[:, e] for e = c, c + grid, ... on CUDA
//     cores (the arithmetic of the router's decode-size kernel) and stores
//     each logit together with the launch's tag in one 64-bit word; every
//     CTA then reads all T x E words, polling (bounded) until each carries
//     the tag. No grid barrier: the tag is the launch number, which each CTA
//     learns from its arrival on a launch counter at its start.
//  B  routing: full-pool top-k and mass when wanted, Eq. 12 on the device,
//     prefix top-k and renormalised weights. For a few tokens every CTA
//     routes all of them itself (no second exchange); for more, each token is
//     routed by one CTA and the picks are exchanged through a second grid
//     barrier. Every CTA then forms the stable dispatch in shared memory; CTA
//     0 writes the intermediates to the workspace.
//  C  experts, as k_ffn_ws: the work list is every gate/up tile (128 weight
//     rows of one active expert) then every down tile, round robin over the
//     CTAs; gate/up tiles take all T token rows of x as the MMA's N operand
//     and store the expert's rows of h; down tiles wait (bounded) for their
//     expert's h, then store the expert's rows of y.
//  D  combine: after storing its y rows a down tile counts, per token and
//     128-feature block, how many of the token's k slots are done; the tile
//     that completes a (token, block) pair sums that pair's k slot rows in
//     slot order (+ residual) into out, with the combine kernel's arithmetic.
// Counters live in the caller's workspace and every launch leaves them at
// zero: the grid barrier (distributed routing only) bumps a generation, the
// launch counter's arrivals return to zero when the last CTA arrives (its
// launch number goes up by one), an expert's readiness count
// is reset by the last of its down tiles, and a (token, block) count by the
// tile that completes it. The first launch on a workspace may find anything
// there: the launch counter carries a 24-bit signature, and an arrival that
// finds it missing (a fresh workspace, or one a timed-out launch marked as
// such) makes CTA 0 clear every counter and the tagged logits and write the
// signature back (release); the other CTAs wait for it (acquire) and arrive
// again. Tags are launch number + 1, never 0, so cleared words never pass
// for logits; the launch number is 24 bits wide, and its wrap carries into
// the signature, which re-initialises the block, so no tag recurs while
// older words can still be read.
#include <type_traits>

#include "route_common.cuh"

namespace decomoe {

constexpr int DL_MIN_T = 1;                // tokens per launch
constexpr int DL_MAX_T = 32;
constexpr int DL_MAX_ROWS = 256;           // routed rows T * k
constexpr int DL_BN = 32;                  // token columns of a tile (MMA N, TMA box rows)
constexpr int DL_BM = 128, DL_BK = 64;     // weight rows per tile, k-block
constexpr int DL_THREADS = 256;            // TMA warp, MMA warp, four epilogue warps, two more for routing
constexpr int DL_FB = 128;                 // features per combine block (= down tile rows)
constexpr int DL_LOCAL_ROUTE_T = 12;       // up to this many tokens every CTA routes them all itself
constexpr uint32_t DL_BULK_CHUNK = 32768;  // bytes per bulk copy of the token rows
constexpr int DL_QN = 4;                   // work items the TMA warp may publish ahead of the MMA and epilogue

// int32 slots of the counter block (the same for every T of a layer shape):
// [0, 2) spare, [2] grid barrier word, [3] work-item counter, [4, 6) launch counter
// (u64: signature in bits 40-63, launch number in bits 16-39, arrivals in
// bits 0-15), [6, 8) spare, then ready[E], done[E] (down tiles finished per
// expert), comb[DL_MAX_T * d / 128], the full-pool picks and weights of the
// distributed routing [2][DL_MAX_ROWS], and the tagged logits
// [DL_MAX_T][E] (u64: logit bits low, tag high).
constexpr int DL_SYNC_HEAD = 8;
constexpr uint64_t DL_SIGNATURE = 0xD3C0AEull;  // 24 bits
__host__ __device__ constexpr int dl_sync_tagged_offset(int E, int d) {
  return DL_SYNC_HEAD + 2 * E + DL_MAX_T * (d / DL_FB) + 2 * DL_MAX_ROWS;
}

struct DlArgs {
  const uint4* x;  // [T, d] bf16
  const uint4* w_r;  // [E, d] bf16
  const float* bias;  // [E] or null
  const uint4* residual;  // [T, d] bf16 or null
  uint4* out;  // [T, d] bf16
  uint4* text_out;  // [T - nv, d] bf16 or null: out without rows [v0, v0 + nv)
  int64_t v0, nv;
  int T, d, E, k, m;
  int K_fixed;  // > 0: prefix length; -1: Eq. 12 on the device
  double p;
  int want_mass;
  float* logits;
  int32_t* topk_idx;
  float* topk_w;
  double* mass;
  int32_t* counts;
  int32_t* offsets;
  int32_t* perm;
  int32_t* inv;
  uint4* x_perm;
  __nv_bfloat16* h;
  __nv_bfloat16* y;
  int32_t* K_dev;
  int32_t* sync;
  int32_t* status;
  uint64_t limit_ns;
};

template <int STAGES>
struct DlCfg {
  static constexpr int A_BYTES = DL_BM * DL_BK * 2;
  static constexpr int B_BYTES = DL_BN * DL_BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * DL_BN;
  static constexpr int NBARS = 2 * STAGES + 6 + 2 * DL_QN;
  static constexpr int XCH_BYTES = 2 * 2 * 32 * 32 * 4;   // SwiGLU up values, double-buffered
  static constexpr int STILE_BYTES = 2 * 32 * DL_BM * 2;  // [2][32 columns][128 features] bf16
  static constexpr int MAXE = DECOMOE_MAX_E;
  // routing state: picks and weights (prefix and full pool), mass, counts,
  // offsets, perm, inv, first work item per expert (two lists)
  static constexpr int ROUTE_BYTES = DL_MAX_ROWS * 4 * 6 + MAXE * 8 + (MAXE + 1) * 4 * 4 + MAXE * 4 + 64 * 4;
  static constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + XCH_BYTES + STILE_BYTES +
                                 NBARS * 8 + ROUTE_BYTES + 64;
};

// dynamic shared memory budget: the per-block maximum less room for the
// kernel's static arrays
constexpr size_t DL_DYN_SMEM_MAX = 232448 - 2048;
template <int S>
constexpr int dl_max_stages_from() {
  return DlCfg<S>::SMEM <= DL_DYN_SMEM_MAX ? S : dl_max_stages_from<S - 1>();
}
template <>
constexpr int dl_max_stages_from<1>() {
  return 1;
}
constexpr int DL_STAGES = dl_max_stages_from<12>();

__device__ __forceinline__ uint64_t ld_acquire_u64(const void* p) {
  uint64_t v;
  asm volatile("ld.acquire.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u64(void* p, uint64_t v) {
  asm volatile("st.release.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
// 1-D bulk copy global -> shared (16-byte aligned, size a multiple of 16),
// completion counted on the mbarrier
__device__ __forceinline__ void bulk_load_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}
__device__ __forceinline__ uint64_t ld_relaxed_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
// two adjacent words (16-byte aligned), each read single-copy atomically
__device__ __forceinline__ void ld_relaxed_u64x2(const uint64_t* p, uint64_t& a, uint64_t& b) {
  asm volatile("ld.relaxed.gpu.global.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(p) : "memory");
}
__device__ __forceinline__ void st_relaxed_u64(uint64_t* p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint64_t atom_add_acquire_u64(uint64_t* p, uint64_t v) {
  uint64_t old;
  asm volatile("atom.acquire.gpu.global.add.u64 %0, [%1], %2;" : "=l"(old) : "l"(p), "l"(v) : "memory");
  return old;
}
__device__ __forceinline__ void red_add_relaxed_u64(uint64_t* p, uint64_t v) {
  asm volatile("red.relaxed.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t atom_add_acq_rel_u32(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ void red_add_release_u32(uint32_t* p, uint32_t v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void red_add_release_s32(int32_t* p, int32_t v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ int atom_add_acq_rel_s32(int32_t* p, int32_t v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// fp32 sum of one bf16 vector scaled by w into acc (the combine's order).
__device__ __forceinline__ void dl_acc_vec(float* acc, const uint4& v, float w) {
  acc[0] = fmaf(w, bf16_lo(v.x), acc[0]);
  acc[1] = fmaf(w, bf16_hi(v.x), acc[1]);
  acc[2] = fmaf(w, bf16_lo(v.y), acc[2]);
  acc[3] = fmaf(w, bf16_hi(v.y), acc[3]);
  acc[4] = fmaf(w, bf16_lo(v.z), acc[4]);
  acc[5] = fmaf(w, bf16_hi(v.z), acc[5]);
  acc[6] = fmaf(w, bf16_lo(v.w), acc[6]);
  acc[7] = fmaf(w, bf16_hi(v.w), acc[7]);
}

// TMAX: the most tokens this form takes (8, 16 or DL_MAX_T): the router's
// per-thread token accumulators, and (up to DL_LOCAL_ROUTE_T) no code for the
// distributed routing. Code run once per launch is fetched cold, so the
// few-token forms run the short versions (measured: T=8 54.6 -> 51.5 us).
template <int STAGES, int TMAX>
__global__ void __launch_bounds__(DL_THREADS, 1)
    k_decode_layer(const __grid_constant__ CUtensorMap tma_w1, const __grid_constant__ CUtensorMap tma_x1,
                   const __grid_constant__ CUtensorMap tma_w2, const __grid_constant__ CUtensorMap tma_x2,
                   const DlArgs g) {
  using C = DlCfg<STAGES>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ float s_red[4][DL_MAX_T];
  __shared__ int s_flag[4];  // [0] counters usable, [1] K, [2] finisher count, [3] the launch's tag (0: not yet)
  __shared__ int s_fin[DL_BN];
  __shared__ int s_q[DL_QN];  // work items in the order this CTA takes them (-1: no more)
  __shared__ int s_qt_store;   // the epilogue's current item
  volatile int* const s_qt = &s_qt_store;
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sA = raw + pad;
  const uint32_t sB = sA + STAGES * C::A_BYTES;
  float* xch = reinterpret_cast<float*>(smem + STAGES * C::STAGE_BYTES);
  __nv_bfloat16* stile = reinterpret_cast<__nv_bfloat16*>(smem + STAGES * C::STAGE_BYTES + C::XCH_BYTES);
  uint64_t* bars =
      reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES + C::XCH_BYTES + C::STILE_BYTES);
  int* s_idx = reinterpret_cast<int*>(bars + C::NBARS);  // [T*k] prefix picks
  float* s_w = reinterpret_cast<float*>(s_idx + DL_MAX_ROWS);
  int* s_fidx = reinterpret_cast<int*>(s_w + DL_MAX_ROWS);  // full-pool picks (mass)
  float* s_fw = reinterpret_cast<float*>(s_fidx + DL_MAX_ROWS);
  int* s_perm = reinterpret_cast<int*>(s_fw + DL_MAX_ROWS);
  int* s_inv = s_perm + DL_MAX_ROWS;
  double* s_mass = reinterpret_cast<double*>(s_inv + DL_MAX_ROWS);
  int* s_cnt = reinterpret_cast<int*>(s_mass + C::MAXE);
  int* s_off = s_cnt + (C::MAXE + 1);
  int* s_tt1 = s_off + (C::MAXE + 1);
  int* s_tt2 = s_tt1 + (C::MAXE + 1);
  uint32_t* s_tmask = reinterpret_cast<uint32_t*>(s_tt2 + (C::MAXE + 1));  // [E] tokens that picked each prefix expert
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(s_tmask + C::MAXE);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tid = threadIdx.x;
  const uint32_t bar0 = smem_u32(bars);
#define FULL_BAR(s) (bar0 + 8u * (s))
#define EMPTY_BAR(s) (bar0 + 8u * (STAGES + (s)))
#define TFULL_BAR(a) (bar0 + 8u * (2 * STAGES + (a)))
#define TEMPTY_BAR(a) (bar0 + 8u * (2 * STAGES + 2 + (a)))
#define DRAIN_BAR (bar0 + 8u * (2 * STAGES + 4))
#define XROWS_BAR (bar0 + 8u * (2 * STAGES + 5))
#define QFULL_BAR(q) (bar0 + 8u * (2 * STAGES + 6 + (q)))
#define QEMPTY_BAR(q) (bar0 + 8u * (2 * STAGES + 6 + DL_QN + (q)))

  const int T = g.T, E = g.E, k = g.k, d = g.d;
  const int N = T * k;
  const int nfb = d / DL_FB;
  uint32_t* const bar_word = reinterpret_cast<uint32_t*>(g.sync + 2);
  uint64_t* const lcount = reinterpret_cast<uint64_t*>(g.sync + 4);
  int32_t* const ready = g.sync + DL_SYNC_HEAD;
  int32_t* const done = ready + E;
  int32_t* const comb = done + E;
  uint64_t* const tagged = reinterpret_cast<uint64_t*>(g.sync + dl_sync_tagged_offset(E, d));  // [T][E] used
  // a timed-out wait: the status says so, and the missing signature makes the
  // next launch re-initialise the counter block
  auto fail = [&]() {
    report_status(g.status, DECOMOE_ERR_TIMEOUT);
    st_relaxed_u64(lcount, 0u);
  };

  if (tid == 0) {
    *s_abort = 0;
    s_flag[3] = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(FULL_BAR(s), 1);
      mbar_init(EMPTY_BAR(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(TFULL_BAR(a), 1);
      mbar_init(TEMPTY_BAR(a), 128);
    }
    mbar_init(DRAIN_BAR, 1);
    mbar_init(XROWS_BAR, 1);
    for (int q = 0; q < DL_QN; ++q) {
      mbar_init(QFULL_BAR(q), 1);
      mbar_init(QEMPTY_BAR(q), 2);  // the MMA thread and the epilogue
    }
    fence_mbar_init();
  }
  // the accumulators' tensor memory, held to the end (every return below
  // frees it first)
  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<uint32_t*>(s_tmem)), C::TMEM_COLS);
    tmem_relinquish();
  } else if (warp == 5 && lane == 0) {
    tma_prefetch_desc(&tma_w1);
    tma_prefetch_desc(&tma_x1);
    tma_prefetch_desc(&tma_w2);
    tma_prefetch_desc(&tma_x2);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  // leave early (a timed-out wait): free the tensor memory first
  auto leave = [&]() {
    if (warp == 1) tmem_dealloc(tmem_base, C::TMEM_COLS);
  };
  // the previous kernel on the stream (which may have used this workspace)
  // has completed and its writes are visible
  pdl_wait();

  // ---------------------------------------------------------------- A: router
  // logits[t, e] = sum_j x[t, j] w_r[e, j] + bias[e] with the router's
  // decode-size arithmetic: threads 0..127 split the row's 16-byte vectors
  // (thread i takes i, i + 128, ...), warp shuffles, then the four warps in
  // order. The T token rows are staged in shared memory first (the TMA ring,
  // unused until the expert phase), all copies in flight at once. Warps 0-3
  // compute; warp 4 meanwhile learns the launch's tag.
  const int vpr = d / 8;
  const uint4* s_x = reinterpret_cast<const uint4*>(smem);
  // the first router row's loads go out with the staging copies (d <= 2048:
  // one pass of GEMV_VPT vectors per thread)
  uint4 wv0[GEMV_VPT];
  const bool pre_w = vpr <= GEMV_THREADS * GEMV_VPT && static_cast<int>(blockIdx.x) < E && tid < GEMV_THREADS;
  // the first router row's bias too (read after the products otherwise)
  const float b0 = (tid < T && g.bias != nullptr && static_cast<int>(blockIdx.x) < E) ? __ldg(g.bias + blockIdx.x) : 0.f;
  if (pre_w) {
#pragma unroll
    for (int i = 0; i < GEMV_VPT; ++i) {
      const int c = tid + GEMV_THREADS * i;
      wv0[i] = (c < vpr) ? __ldg(g.w_r + static_cast<int64_t>(blockIdx.x) * vpr + c) : make_uint4(0u, 0u, 0u, 0u);
    }
  }
  if (tid == 0) {
    // the T rows in bulk copies, completion counted on one barrier
    const uint32_t bytes = static_cast<uint32_t>(T) * static_cast<uint32_t>(vpr) * 16u;
    mbar_arrive_expect_tx(XROWS_BAR, bytes);
    for (uint32_t off = 0; off < bytes; off += DL_BULK_CHUNK)
      bulk_load_g2s(sA + off, reinterpret_cast<const uint8_t*>(g.x) + off,
                    bytes - off < DL_BULK_CHUNK ? bytes - off : DL_BULK_CHUNK, XROWS_BAR);
  }
  volatile int* const vflag = s_flag;
  if (tid < GEMV_THREADS) {
    if (!mbar_wait(XROWS_BAR, 0, g.limit_ns, s_abort)) fail();
    for (int e = blockIdx.x; e < E; e += gridDim.x) {
      const uint4* wr = g.w_r + static_cast<int64_t>(e) * vpr;
      float acc[TMAX];
#pragma unroll
      for (int j = 0; j < TMAX; ++j) acc[j] = 0.f;
      for (int c0 = 0; c0 < vpr; c0 += GEMV_THREADS * GEMV_VPT) {
        uint4 wv[GEMV_VPT];
#pragma unroll
        for (int i = 0; i < GEMV_VPT; ++i) {
          const int c = c0 + tid + GEMV_THREADS * i;
          wv[i] = (pre_w && e == static_cast<int>(blockIdx.x)) ? wv0[i]
                  : (c < vpr)                                  ? __ldg(wr + c)
                                                               : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int i = 0; i < GEMV_VPT; ++i) {
          const int c = c0 + tid + GEMV_THREADS * i;
          if (c < vpr) {
#pragma unroll
            for (int j = 0; j < TMAX; ++j)
              if (j < T) acc[j] = dot8_bf16(wv[i], s_x[j * vpr + c], acc[j]);
          }
        }
      }
#pragma unroll
      for (int j = 0; j < TMAX; ++j) {
        if (j < T) {
          float v = acc[j];
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
          if (lane == 0) s_red[warp][j] = v;
        }
      }
      named_bar_sync(2, GEMV_THREADS);
      if (tid < T) {
        float v = s_red[0][tid];
#pragma unroll
        for (int w = 1; w < GEMV_THREADS / 32; ++w) v += s_red[w][tid];
        v += g.bias == nullptr ? 0.f : e == static_cast<int>(blockIdx.x) ? b0 : __ldg(g.bias + e);
        // the logit and the launch's tag in one single-copy-atomic word
        int tg = vflag[3];
        if (tg == 0) {
          const uint64_t t0 = globaltimer_ns();
          while (tg == 0 && !*s_abort && globaltimer_ns() - t0 <= g.limit_ns) tg = vflag[3];
        }
        if (tg != 0)
          st_relaxed_u64(tagged + tid * E + e,
                         (static_cast<uint64_t>(static_cast<uint32_t>(tg)) << 32) | __float_as_uint(v));
      }
      named_bar_sync(2, GEMV_THREADS);
    }
  } else if (warp == GEMV_THREADS / 32) {
    // Arrive on the launch counter: the launch number in the returned word is
    // this launch's for every CTA (the round cannot complete before all of
    // them have arrived), and the last arrival moves it to the next number.
    // Without the signature, CTA 0 (re)initialises the counter block and the
    // other CTAs wait for that, then arrive again.
    const uint32_t G = gridDim.x;
    uint64_t old = 0;
    if (lane == 0) old = atom_add_acquire_u64(lcount, 1u);
    old = __shfl_sync(0xffffffffu, old, 0);
    bool ok = true;
    if ((old >> 40) != DL_SIGNATURE) {
      if (blockIdx.x == 0) {
        // the barrier word, the work-item counter, ready, done, comb, the
        // distributed picks and the tagged logits, then the signature
        // (launch 0, no arrivals)
        const int n = dl_sync_tagged_offset(E, d) + 2 * DL_MAX_T * E;
        g.sync[2] = 0;
        g.sync[3] = 0;
        for (int i = DL_SYNC_HEAD + lane; i < n; i += 32) g.sync[i] = 0;
        __syncwarp();
        if (lane == 0) {
          __threadfence();
          st_release_u64(lcount, DL_SIGNATURE << 40);
          old = atom_add_acquire_u64(lcount, 1u);
        }
      } else if (lane == 0) {
        const uint64_t t0 = globaltimer_ns();
        while ((ld_acquire_u64(lcount) >> 40) != DL_SIGNATURE)
          if (globaltimer_ns() - t0 > g.limit_ns) {
            ok = false;
            break;
          }
        if (ok) old = atom_add_acquire_u64(lcount, 1u);
      }
    }
    if (lane == 0) {
      if (ok && (old >> 40) == DL_SIGNATURE) {
        if ((old & 0xFFFFu) == G - 1u) red_add_relaxed_u64(lcount, 0x10000u - G);
        vflag[3] = static_cast<int>(static_cast<uint32_t>((old >> 16) & 0xFFFFFFu) + 1u);  // never 0
      } else {
        *s_abort = 1;
        fail();
      }
    }
  }

  // ---------------------------------------------------------------- grid barrier
  // (distributed routing only) One word: arrivals in the low 16 bits, a
  // generation in the high bits. The last arrival (acquire-release, after
  // every CTA's writes) adds 0x10000 - grid, which empties the count and
  // bumps the generation.
  auto grid_sync = [&]() -> bool {
    __syncthreads();
    if (tid == 0) {
      bool ok = true;
      const uint64_t t0 = globaltimer_ns();
      const uint32_t G = gridDim.x;
      const uint32_t old = atom_add_acq_rel_u32(bar_word, 1u);
      if ((old & 0xFFFFu) == G - 1u) {
        red_add_release_u32(bar_word, 0x10000u - G);
      } else {
        // short sleeps between polls keep the waiting CTAs' loads off the
        // word the last arrival has to update
        while ((ld_acquire_u32(bar_word) >> 16) == (old >> 16)) {
          __nanosleep(64);
          if (globaltimer_ns() - t0 > g.limit_ns) {
            ok = false;
            break;
          }
        }
      }
      s_flag[0] = ok;
      if (!ok) fail();
    }
    __syncthreads();
    return s_flag[0] != 0;
  };
  // every thread past the router (the ring's x rows are no longer read)
  __syncthreads();
  if (*s_abort) {
    leave();
    return;
  }
  const uint32_t tag = static_cast<uint32_t>(s_flag[3]);

  // ---------------------------------------------------------------- B: routing
  // Up to DL_LOCAL_ROUTE_T tokens every CTA routes them all itself (same
  // inputs, same arithmetic: the same result everywhere) from the logits
  // staged in shared memory, one warp per token. Above that (fixed prefix
  // only) CTA t routes token t, publishes its picks, and a second grid
  // barrier precedes the dispatch. Lane l holds logits l, l+32, ...
  const int Kd = g.K_fixed > 0 ? g.K_fixed : E;  // expert groups of the dispatch
  // one token per CTA, then a second barrier (never in the few-token forms)
  const bool dist = TMAX > DL_LOCAL_ROUTE_T && T > DL_LOCAL_ROUTE_T;
  float* s_lg = reinterpret_cast<float*>(smem);  // [T][E], in the ring
  float* s_wt = s_lg + T * E;                     // [T][E] full-pool pick weights (0: not picked)
  int32_t* const g_fpick = comb + DL_MAX_T * nfb;  // [T*k] full-pool picks (distributed routing)
  float* const g_fpw = reinterpret_cast<float*>(g_fpick + N);
  {
    for (int i = tid; i < T * E / 4; i += DL_THREADS)
      reinterpret_cast<float4*>(s_wt)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i = tid; i < C::MAXE; i += DL_THREADS) s_tmask[i] = 0u;
    if (!dist) {
      // every logit, once its word carries this launch's tag (pairs of
      // words, up to four pairs per thread in flight per round; bounded)
      bool ok = true;
      uint64_t t0 = 0;  // the clock is read once a round finds words missing
      const int npair = T * E / 2;  // E is a multiple of 4
      for (int i0 = 0; ok && i0 < npair; i0 += 4 * DL_THREADS) {
        uint64_t w[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) w[j] = 0u;  // tag 0: not read yet
        for (;;) {
          // (re)read the pairs not complete yet
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int i = i0 + tid + DL_THREADS * j;
            if (i >= npair) {
              w[2 * j] = w[2 * j + 1] = static_cast<uint64_t>(tag) << 32;
            } else if (static_cast<uint32_t>(w[2 * j] >> 32) != tag || static_cast<uint32_t>(w[2 * j + 1] >> 32) != tag) {
              ld_relaxed_u64x2(tagged + 2 * i, w[2 * j], w[2 * j + 1]);
            }
          }
          bool pend = false;
#pragma unroll
          for (int j = 0; j < 8; ++j) pend |= static_cast<uint32_t>(w[j] >> 32) != tag;
          if (!pend) break;
          if (t0 == 0) t0 = globaltimer_ns();
          if (*s_abort || globaltimer_ns() - t0 > g.limit_ns) {
            ok = false;
            break;
          }
          __nanosleep(64);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int i = i0 + tid + DL_THREADS * j;
          if (i < npair) {
            s_lg[2 * i] = __uint_as_float(static_cast<uint32_t>(w[2 * j]));
            s_lg[2 * i + 1] = __uint_as_float(static_cast<uint32_t>(w[2 * j + 1]));
          }
        }
      }
      if (!ok) {
        *s_abort = 1;
        fail();
      }
    }
  }
  __syncthreads();
  if (*s_abort) {
    leave();
    return;
  }
  if (!dist && blockIdx.x == 0)
    for (int i = tid; i < T * E; i += DL_THREADS) g.logits[i] = s_lg[i];
  if (dist) {
    // CTA t < T routes token t (warp 0; fixed prefix) and publishes its picks
    if (static_cast<int>(blockIdx.x) < T && warp == 0) {
      const int t = blockIdx.x;
      const uint64_t* row = tagged + t * E;
      const int lim = g.want_mass ? E : g.K_fixed;
      // row t, once each word carries this launch's tag (bounded; on time-out
      // the status says so and the launch goes on with what it read)
      float lv[8];
      {
        const uint64_t t0 = globaltimer_ns();
        uint64_t wv[8];
        for (;;) {
          bool pend = false;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int e = lane + 32 * i;
            wv[i] = e < E ? ld_relaxed_u64(row + e) : static_cast<uint64_t>(tag) << 32;
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) pend |= static_cast<uint32_t>(wv[i] >> 32) != tag;
          if (!__any_sync(0xffffffffu, pend)) break;
          if (__any_sync(0xffffffffu, globaltimer_ns() - t0 > g.limit_ns)) {  // warp-uniform exit
            if (lane == 0) fail();
            break;
          }
          __nanosleep(64);
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int e = lane + 32 * i;
          lv[i] = __uint_as_float(static_cast<uint32_t>(wv[i]));
          if (e < E) g.logits[t * E + e] = lv[i];
        }
      }
      uint32_t v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int e = lane + 32 * i;
        v[i] = (e < lim) ? fkey(lv[i]) : 0u;
      }
      float my_v;
      int my_i;
      warp_topk(v, lim, k, lane, my_v, my_i);
      if (g.want_mass) {
        const float wf = pick_weight(my_v, lane, k);
        if (lane < k) {
          g_fpick[t * k + lane] = my_i;
          g_fpw[t * k + lane] = wf;
        }
        const bool inside = __all_sync(0xffffffffu, lane >= k || my_i < g.K_fixed);
        if (!inside) warp_topk(v, g.K_fixed, k, lane, my_v, my_i);
      }
      const float w = pick_weight(my_v, lane, k);
      if (lane < k) {
        g.topk_idx[t * k + lane] = my_i;
        g.topk_w[t * k + lane] = w;
      }
    }
    if (!grid_sync()) {
      leave();
      return;
    }
    for (int f = tid; f < N; f += DL_THREADS) {
      const int t = f / k;
      const int e = __ldcg(g.topk_idx + f);
      s_idx[f] = e;
      s_w[f] = __ldcg(g.topk_w + f);
      atomicOr(&s_tmask[e], 1u << t);
      if (g.want_mass) {
        const int fe = __ldcg(g_fpick + f);
        const float fw = __ldcg(g_fpw + f);
        s_fidx[f] = fe;
        s_fw[f] = fw;
        s_wt[t * E + fe] = fw;
      }
    }
    __syncthreads();
  }
  // one routing pass; NSL key slots per lane (4 cover up to 128 experts).
  // The full pool's picks (with the mass) and the prefix picks come from one
  // loop body, so its code is fetched once for both rounds.
  auto route_tokens = [&](auto nsl, int lim_fixed, bool full) {
    constexpr int NSL = decltype(nsl)::value;
    // full: picks over [0, E) into s_fidx / s_fw, then, with a fixed prefix,
    // the prefix picks; else picks over [0, lim_fixed)
    const int Kp = full ? g.K_fixed : lim_fixed;
    for (int t = warp; t < T; t += DL_THREADS / 32) {
      const float* row = s_lg + t * E;
      uint32_t v[NSL];
#pragma unroll
      for (int i = 0; i < NSL; ++i) {
        const int e = lane + 32 * i;
        v[i] = (e < E) ? fkey(row[e]) : 0u;
      }
      float my_v = 0.f;
      int my_i = 0;
      for (int r = full ? 0 : 1; r < 2; ++r) {
        if (r == 1 && Kp <= 0) break;  // the prefix is chosen after the mass
        // full-pool picks all inside the prefix are the prefix picks too
        const bool reuse = r == 1 && full && __all_sync(0xffffffffu, lane >= k || my_i < Kp);
        if (!reuse) warp_topk_n<NSL>(v, r == 0 ? E : Kp, k, lane, my_v, my_i);
        const float w = pick_weight(my_v, lane, k);
        if (lane < k) {
          if (r == 0) {
            s_fidx[t * k + lane] = my_i;
            s_fw[t * k + lane] = w;
            s_wt[t * E + my_i] = w;
          } else {
            s_idx[t * k + lane] = my_i;
            s_w[t * k + lane] = w;
            atomicOr(&s_tmask[my_i], 1u << t);
          }
        }
      }
    }
  };
  auto route_pass = [&](int lim_fixed, bool full) {
    if (E <= 128)
      route_tokens(std::integral_constant<int, 4>(), lim_fixed, full);
    else
      route_tokens(std::integral_constant<int, 8>(), lim_fixed, full);
  };
  // At most two passes from one call site (code run once per launch is
  // fetched cold): pass 0 the full pool (with the mass) or the fixed prefix,
  // then Eq. 11's mass, and with the prefix selected on the device (Eq. 12)
  // pass 1 over [0, K).
  for (int pass = 0; pass < 2; ++pass) {
    if (pass == 1) {
      if (g.want_mass) {
        // Eq. 11 as the routing kernels form it: fp32 sums per block of 8
        // tokens in token order (a token picks an expert at most once; the
        // table's zeros add nothing), then the fixed fp64 tree over the blocks
        for (int e = tid; e < E; e += DL_THREADS) {
          float a[4] = {0.f, 0.f, 0.f, 0.f};  // blocks of 8 tokens (T <= 32)
#pragma unroll
          for (int b = 0; b < 4; ++b)
            for (int tt = 8 * b; tt < T && tt < 8 * b + 8; ++tt) a[b] += s_wt[tt * E + e];
          const double me = T <= 8 ? static_cast<double>(a[0])
                                   : (static_cast<double>(a[0]) + static_cast<double>(a[2])) +
                                         (static_cast<double>(a[1]) + static_cast<double>(a[3]));
          s_mass[e] = me;
          if (blockIdx.x == 0) g.mass[e] = me;
        }
      }
      if (g.K_fixed >= 0) break;
      __syncthreads();
      if (tid == 0) {
        s_flag[1] = select_prefix_seq(s_mass, E, k, g.p);
        if (blockIdx.x == 0) *g.K_dev = s_flag[1];
      }
      __syncthreads();
    } else if (dist) {
      continue;  // the picks were routed per CTA and exchanged above
    }
    const bool full = pass == 0 && g.want_mass;
    route_pass(pass == 1 ? s_flag[1] : (full ? 0 : g.K_fixed), full);
    __syncthreads();
  }
  __syncthreads();
  // dispatch: counts and exclusive offsets from the per-expert token masks;
  // the stable rank of pair f = t*k + j is the number of earlier tokens that
  // picked its expert (a token picks an expert at most once)
  const int nwb1 = 2 * g.m / DL_BM, nwb2 = d / DL_BM;
  if (warp < 2) {
    const int per = (Kd + 31) / 32;  // <= 8
    int cnt[8];
    int run = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e = lane * per + i;
      cnt[i] = (i < per && e < Kd) ? (warp == 0 ? __popc(s_tmask[e]) : (s_tmask[e] != 0u ? 1 : 0)) : 0;
      run += cnt[i];
    }
    int incl = run;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    int acc = incl - run;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e = lane * per + i;
      if (i < per && e < Kd) {
        if (warp == 0) {
          s_off[e] = acc;
          s_cnt[e] = cnt[i];
        } else {
          // work list: items per expert with rows (one token chunk: T <= 32)
          s_tt1[e] = acc * nwb1;
          s_tt2[e] = acc * nwb2;
        }
        acc += cnt[i];
      }
    }
    if (lane == 31) {
      if (warp == 0) {
        s_off[Kd] = incl;
      } else {
        s_tt1[Kd] = incl * nwb1;
        s_tt2[Kd] = incl * nwb2;
      }
    }
  }
  __syncthreads();
  for (int f = tid; f < N; f += DL_THREADS) {
    const int e = s_idx[f];
    const int t = f / k;
    const int r = s_off[e] + __popc(s_tmask[e] & ((1u << t) - 1u));
    s_perm[r] = t;
    s_inv[f] = r;
  }
  __syncthreads();
  if (blockIdx.x == 0) {
    for (int f = tid; f < N; f += DL_THREADS) {
      if (!dist) {
        g.topk_idx[f] = s_idx[f];
        g.topk_w[f] = s_w[f];
      }
      g.inv[f] = s_inv[f];
      g.perm[f] = s_perm[f];
    }
    for (int e = tid; e < Kd; e += DL_THREADS) {
      g.counts[e] = s_cnt[e];
      g.offsets[e] = s_off[e];
    }
    if (tid == 0) g.offsets[Kd] = s_off[Kd];
  }
  // the ring held x and the logits (generic proxy); TMA writes it from here on
  fence_proxy_async_smem();
  const int total1 = s_tt1[Kd], total = total1 + s_tt2[Kd];

  // ---------------------------------------------------------------- C, D: experts and combine
  __syncthreads();
  // item -> (down?, expert, weight block); expert = last e with s_tt[e] <= i
  auto item = [&](int t, bool& dn, int& eg, int& wb) {
    dn = t >= total1;
    const int* tt = dn ? s_tt2 : s_tt1;
    const int i = dn ? t - total1 : t;
    int lo = 0, hi = Kd - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (tt[mid] <= i)
        lo = mid;
      else
        hi = mid - 1;
    }
    // experts without rows share their successor's first item: take the last
    // expert whose range is non-empty
    eg = lo;
    wb = i - tt[lo];
  };

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0)
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    uint32_t armed = 0, armed_ph = 0;
    const uint64_t pol_once = policy_evict_first();  // every weight block is read once per step
    // Work items: the first is this CTA's index, every later one comes from
    // the shared counter (item grid + n for the n-th draw), drawn once the
    // current item's last load is out (the draw's round trip hides behind
    // the loads in flight), so CTAs that finish early take more. Each CTA
    // draws until it gets an index past the list (a CTA without a first item
    // draws once): max(total, grid) draws in all, and the last of them
    // returns the counter to zero for the next launch.
    int32_t* const sched = g.sync + 3;
    const int G = static_cast<int>(gridDim.x);
    const int ndraw = total > G ? total : G;
    auto draw = [&]() -> int {
      const int f = atomicAdd(sched, 1);
      if (f == ndraw - 1) *sched = 0;
      return G + f;
    };
    int t = blockIdx.x;
    for (int n = 0;; ++n) {
      // publish the item (or the end) to the MMA and epilogue warps
      if (lane == 0) {
        const int qs = n % DL_QN;
        if (!mbar_wait(QEMPTY_BAR(qs), ((n / DL_QN) & 1u) ^ 1u, g.limit_ns, s_abort)) {
          ok = false;
        } else {
          s_q[qs] = t < total ? t : -1;
          mbar_arrive(QFULL_BAR(qs));
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      if (t >= total) {
        if (n == 0 && lane == 0) draw();
        break;
      }
      bool dn;
      int eg, wb;
      item(t, dn, eg, wb);
      if (lane == 0) {
        const CUtensorMap* tw = dn ? &tma_w2 : &tma_w1;
        const CUtensorMap* tx = dn ? &tma_x2 : &tma_x1;
        const int wrow0 = eg * (dn ? d : 2 * g.m) + wb * DL_BM;
        const int brow0 = dn ? s_off[eg] : 0;  // h rows of the expert, or all T rows of x
        const int KB = (dn ? g.m : d) / DL_BK;
        int pre = 0;
        if (dn) {
          const int need = nwb1;
          const bool met = ld_acquire_gpu(ready + eg) >= need;
          if (met) {
            fence_proxy_async_all();  // h, written by generic stores, read through the tensor map
          } else {
            // weights first (they depend on nothing), then wait for h
            pre = KB < STAGES ? KB : STAGES;
            const int st0 = stage;
            for (int kb = 0; kb < pre; ++kb) {
              if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
                ok = false;
                break;
              }
              mbar_arrive_expect_tx(FULL_BAR(stage), C::STAGE_BYTES);
              tma_load_2d_hint(sA + stage * C::A_BYTES, tw, FULL_BAR(stage), kb * DL_BK, wrow0, pol_once);
              armed |= 1u << stage;
              armed_ph = (armed_ph & ~(1u << stage)) | (ph << stage);
              if (++stage == STAGES) {
                stage = 0;
                ph ^= 1u;
              }
            }
            if (ok) {
              const volatile int32_t* rp = ready + eg;
              const uint64_t t0 = globaltimer_ns();
              while (*rp < need) {
                if (*s_abort || globaltimer_ns() - t0 > g.limit_ns) {
                  ok = false;
                  break;
                }
              }
              __threadfence();
              fence_proxy_async_all();
            }
            if (ok) {
              int st = st0;
              for (int kb = 0; kb < pre; ++kb) {
                tma_load_2d(sB + st * C::B_BYTES, tx, FULL_BAR(st), kb * DL_BK, brow0);
                if (++st == STAGES) st = 0;
              }
            }
          }
        }
        for (int kb = pre; ok && kb < KB; ++kb) {
          if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(FULL_BAR(stage), C::STAGE_BYTES);
          tma_load_2d_hint(sA + stage * C::A_BYTES, tw, FULL_BAR(stage), kb * DL_BK, wrow0, pol_once);
          tma_load_2d(sB + stage * C::B_BYTES, tx, FULL_BAR(stage), kb * DL_BK, brow0);
          armed |= 1u << stage;
          armed_ph = (armed_ph & ~(1u << stage)) | (ph << stage);
          if (++stage == STAGES) {
            stage = 0;
            ph ^= 1u;
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      const int tn = lane == 0 ? draw() : 0;
      t = __shfl_sync(0xffffffffu, tn, 0);
    }
    if (lane == 0 && !ok) {
      *s_abort = 1;
      fail();
      int no_abort = 0;
      for (int s = 0; s < STAGES; ++s)
        if ((armed >> s) & 1u) mbar_wait(FULL_BAR(s), (armed_ph >> s) & 1u, g.limit_ns, &no_abort);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------ MMA issuer
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true, issued = false;
    for (int it = 0;; ++it) {
      const int qs = it % DL_QN;
      if (!mbar_wait(QFULL_BAR(qs), (it / DL_QN) & 1u, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      const int t = *reinterpret_cast<volatile int*>(&s_q[qs]);
      mbar_arrive(QEMPTY_BAR(qs));
      if (t < 0) break;
      bool dn;
      int eg, wb;
      item(t, dn, eg, wb);
      const int KB = (dn ? g.m : d) / DL_BK;
      const int ncol = dn ? s_off[eg + 1] - s_off[eg] : T;
      const uint32_t idesc = idesc_bf16_f32(DL_BM, (ncol + 15) & ~15);
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait(TEMPTY_BAR(acc), aph ^ 1u, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t dt = tmem_base + static_cast<uint32_t>(acc * DL_BN);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(FULL_BAR(stage), ph, g.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = smem_desc_kmajor<DL_BK>(sA + stage * C::A_BYTES);
        const uint64_t bd = smem_desc_kmajor<DL_BK>(sB + stage * C::B_BYTES);
#pragma unroll
        for (int kk = 0; kk < DL_BK / 16; ++kk)
          tc_mma_f16(dt, ad + 2u * kk, bd + 2u * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
        tc_commit(EMPTY_BAR(stage));
        issued = true;
        if (++stage == STAGES) {
          stage = 0;
          ph ^= 1u;
        }
      }
      if (!ok) break;
      tc_commit(TFULL_BAR(acc));
    }
    if (!ok) {
      *s_abort = 1;
      fail();
      if (issued) {
        int no_abort = 0;
        tc_commit(DRAIN_BAR);
        mbar_wait(DRAIN_BAR, 0, g.limit_ns, &no_abort);
      }
    }
  } else if (warp >= 2 && warp < 6) {
    // ------------------------------------------------ epilogue (4 warps)
    const int q = warp & 3;  // TMEM lanes [32q, 32q + 32)
    const int et = tid - 64;  // 0..127
    // the dispatched rows x_perm[r] = x[perm[r]] (an inspection copy: the
    // expert tiles read x itself), rows r = blockIdx.x + grid * i
    for (int r = blockIdx.x + gridDim.x * (warp - 2); r < N; r += 4 * gridDim.x) {
      const uint4* src = g.x + static_cast<int64_t>(s_perm[r]) * vpr;
      uint4* dst = g.x_perm + static_cast<int64_t>(r) * vpr;
      for (int c = lane; c < vpr; c += 32) dst[c] = __ldg(src + c);
    }
    int xpar = 0;
    bool ok = true;
    for (int it = 0;; ++it) {
      // one thread takes the item from the queue and hands it (or -2 for a
      // wait that gave up) to the other 127 through s_qt
      if (et == 0) {
        const int qs = it % DL_QN;
        if (mbar_wait(QFULL_BAR(qs), (it / DL_QN) & 1u, g.limit_ns, s_abort)) {
          *s_qt = *reinterpret_cast<volatile int*>(&s_q[qs]);
          mbar_arrive(QEMPTY_BAR(qs));
        } else {
          *s_qt = -2;
        }
      }
      named_bar_sync(1, 128);
      const int t = *s_qt;
      if (t == -2) {
        ok = false;
        break;
      }
      if (t < 0) break;
      bool dn;
      int eg, wb;
      item(t, dn, eg, wb);
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait(TFULL_BAR(acc), aph, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t tb = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * DL_BN);
      const int r0 = s_off[eg], nr = s_off[eg + 1] - s_off[eg];
      // accumulator column c: token c of x (gate/up) or row r0 + c of h (down)
      const int OC = dn ? DL_BM : DL_BM / 2;
      uint32_t rr[32];
      tmem_ld32(tb, rr);
      tc_wait_ld();
      __nv_bfloat16* st = stile + xpar * (32 * DL_BM);
      if (!dn) {
        const bool is_gate = q < 2;
        const int pr = q & 1;
        float* xb = xch + (xpar * 2 + pr) * 1024;  // [32 columns][32 lanes]
        if (!is_gate) {
#pragma unroll
          for (int c = 0; c < 32; ++c) xb[c * 32 + lane] = __uint_as_float(rr[c]);
        }
        named_bar_sync(1, 128);
        if (is_gate) {
#pragma unroll
          for (int c = 0; c < 32; ++c)
            st[c * OC + pr * 32 + lane] = __float2bfloat16_rn(silu_f(__uint_as_float(rr[c])) * xb[c * 32 + lane]);
        }
      } else {
#pragma unroll
        for (int c = 0; c < 32; ++c) st[c * OC + q * 32 + lane] = __float2bfloat16_rn(__uint_as_float(rr[c]));
      }
      tc_fence_before();
      mbar_arrive(TEMPTY_BAR(acc));
      named_bar_sync(1, 128);
      // store the expert's rows: h[r, wb*64 ..] from column perm[r], or
      // y[r, wb*128 ..] from column r - r0
      const int VPR = OC / 8;
      __nv_bfloat16* outp = dn ? g.y : g.h;
      const int64_t ld = dn ? d : g.m;
      for (int v = et; v < nr * VPR; v += 128) {
        const int i = v / VPR, cv = v - i * VPR;
        const int col = dn ? i : s_perm[r0 + i];
        const uint4 val = *reinterpret_cast<const uint4*>(st + col * OC + cv * 8);
        *reinterpret_cast<uint4*>(outp + static_cast<int64_t>(r0 + i) * ld + wb * OC + cv * 8) = val;
      }
      xpar ^= 1;
      if (!dn) {
        // this item's h slice is stored: publish it to the down items of eg
        fence_proxy_async_all();
        named_bar_sync(1, 128);
        if (et == 0) red_add_release_s32(ready + eg, 1);
      } else {
        // y rows of block wb stored: count them per token; the tile that
        // completes a token's k slots of this block combines them
        if (et == 0) s_flag[2] = 0;
        named_bar_sync(1, 128);
        if (et < nr) {
          const int tok = s_perm[r0 + et];
          // release this tile's y rows; the k-th arrival acquires the others'
          const int old = atom_add_acq_rel_s32(comb + tok * nfb + wb, 1);
          if (old == k - 1) {
            // nothing else touches this count in the launch
            comb[tok * nfb + wb] = 0;
            s_fin[atomicAdd(&s_flag[2], 1)] = tok;
          }
        }
        named_bar_sync(1, 128);
        const int nfin = s_flag[2];
        // 16 vectors of 8 features per finished token, 8 tokens per pass
        for (int u = et; u < nfin * (DL_FB / 8); u += 128) {
          const int tok = s_fin[u / (DL_FB / 8)];
          const int cv = wb * (DL_FB / 8) + u % (DL_FB / 8);
          float a8[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) a8[i] = 0.f;
          for (int j = 0; j < k; ++j) {
            const int r = s_inv[tok * k + j];
            const uint4 yv = __ldcg(reinterpret_cast<const uint4*>(g.y) + static_cast<int64_t>(r) * vpr + cv);
            dl_acc_vec(a8, yv, s_w[tok * k + j]);
          }
          if (g.residual != nullptr) dl_acc_vec(a8, __ldg(g.residual + static_cast<int64_t>(tok) * vpr + cv), 1.0f);
          const uint4 o = make_uint4(pack_bf16x2(a8[0], a8[1]), pack_bf16x2(a8[2], a8[3]),
                                     pack_bf16x2(a8[4], a8[5]), pack_bf16x2(a8[6], a8[7]));
          g.out[static_cast<int64_t>(tok) * vpr + cv] = o;
          // the visual-block removal of the output: text rows also go to text_out
          if (g.text_out != nullptr && (tok < g.v0 || tok >= g.v0 + g.nv))
            g.text_out[(tok < g.v0 ? tok : tok - g.nv) * vpr + cv] = o;
        }
        // the last down tile of expert eg resets its readiness count (every
        // down tile of eg has read it before its own loads)
        if (et == 0 && atomicAdd(done + eg, 1) == nwb2 - 1) {
          ready[eg] = 0;
          done[eg] = 0;
        }
      }
    }
    if (!ok) {
      *s_abort = 1;
      fail();
    }
  }
  pdl_trigger();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
#undef FULL_BAR
#undef EMPTY_BAR
#undef TFULL_BAR
#undef TEMPTY_BAR
#undef DRAIN_BAR
#undef XROWS_BAR
#undef QFULL_BAR
#undef QEMPTY_BAR
}

bool decode_layer_supported(int64_t T, int d, int E, int k, int m, int dtype, int K_fixed) {
  // x rows and the logits are staged in the TMA ring during the first phases
  constexpr size_t ring = static_cast<size_t>(DL_STAGES) * DlCfg<DL_STAGES>::STAGE_BYTES;
  return dtype == DECOMOE_BF16 && T >= DL_MIN_T && T <= DL_MAX_T && T * k <= DL_MAX_ROWS &&
         (K_fixed > 0 || (K_fixed == -1 && T <= DL_LOCAL_ROUTE_T)) && E >= 1 &&
         E <= DECOMOE_MAX_E && E % 4 == 0 && k >= 1 && k <= 32 && k <= E && d % 256 == 0 && m % 128 == 0 &&
         static_cast<size_t>(T) * d * 2 <= ring && static_cast<size_t>(T) * E * 8 <= ring;
}

size_t decode_layer_sync_ints(int64_t T, int d, int E) {
  if (T < DL_MIN_T || T > DL_MAX_T) return 0;  // the one-launch layer never runs there
  return align_up(static_cast<size_t>(dl_sync_tagged_offset(E, d) + 2 * DL_MAX_T * E), 64);
}

int launch_decode_layer(const void* x, const void* w_r, const float* bias, const void* w_gate_up, const void* w_down,
                        int64_t T, int d, int E, int k, int m, int K_fixed, double p, const void* residual, void* out,
                        void* text_out, int64_t v0, int64_t nv, float* logits, int32_t* topk_idx, float* topk_w, double* mass, int32_t* counts,
                        int32_t* offsets, int32_t* perm, int32_t* inv, void* x_perm, void* h, void* y, int32_t* K_dev,
                        int32_t* sync, int32_t* status, cudaStream_t s) {
  using C = DlCfg<DL_STAGES>;
  DM_ARG_CHECK(aligned16(x) && aligned16(w_r) && aligned16(w_gate_up) && aligned16(w_down) && aligned16(out) &&
                   (residual == nullptr || aligned16(residual)) && (text_out == nullptr || aligned16(text_out)),
               "moe_layer: bf16 operands must be 16-byte aligned");
  DM_ARG_CHECK((reinterpret_cast<uintptr_t>(sync) & 15u) == 0, "moe_layer: workspace misaligned");
  CUtensorMap tw1, tx1, tw2, tx2;
  DM_RET(make_tmap_bf16(&tw1, w_gate_up, static_cast<uint64_t>(d), static_cast<uint64_t>(E) * 2 * m, DL_BM, DL_BK));
  DM_RET(make_tmap_bf16(&tx1, x, static_cast<uint64_t>(d), static_cast<uint64_t>(T), DL_BN, DL_BK));
  DM_RET(make_tmap_bf16(&tw2, w_down, static_cast<uint64_t>(m), static_cast<uint64_t>(E) * d, DL_BM, DL_BK));
  DM_RET(make_tmap_bf16(&tx2, h, static_cast<uint64_t>(m), static_cast<uint64_t>(T) * k, DL_BN, DL_BK));
  DlArgs g;
  g.x = static_cast<const uint4*>(x);
  g.w_r = static_cast<const uint4*>(w_r);
  g.bias = bias;
  g.residual = static_cast<const uint4*>(residual);
  g.out = static_cast<uint4*>(out);
  g.text_out = static_cast<uint4*>(text_out);
  g.v0 = v0;
  g.nv = nv;
  g.T = static_cast<int>(T);
  g.d = d;
  g.E = E;
  g.k = k;
  g.m = m;
  g.K_fixed = K_fixed;
  g.p = p;
  g.want_mass = (K_fixed == -1 || p > 0.0) ? 1 : 0;
  g.logits = logits;
  g.topk_idx = topk_idx;
  g.topk_w = topk_w;
  g.mass = mass;
  g.counts = counts;
  g.offsets = offsets;
  g.perm = perm;
  g.inv = inv;
  g.x_perm = static_cast<uint4*>(x_perm);
  g.h = static_cast<__nv_bfloat16*>(h);
  g.y = static_cast<__nv_bfloat16*>(y);
  g.K_dev = K_dev;
  g.sync = sync;
  g.status = status;
  g.limit_ns = static_cast<uint64_t>(wait_limit_ns());
  auto kern = T <= 8    ? k_decode_layer<DL_STAGES, 8>
              : T <= 16 ? k_decode_layer<DL_STAGES, 16>
                        : k_decode_layer<DL_STAGES, DL_MAX_T>;
  static_assert(C::SMEM <= DL_DYN_SMEM_MAX, "shared memory budget");
  static_assert(C::SMEM > 232448 / 2, "one CTA per SM: the grid barrier needs every CTA resident");
  DM_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(C::SMEM)));
  DM_CUDA_CHECK(launch_pdl(kern, dim3(sm_count()), dim3(DL_THREADS), C::SMEM, s, tw1, tx1, tw2, tx2, g));
  return DECOMOE_OK;
}

}  // namespace decomoe
