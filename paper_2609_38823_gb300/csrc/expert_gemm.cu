// Grouped expert GEMMs of the prefix-MoE layer (DecoMoE Algorithm 2: evaluate
// only the first K physically contiguous expert MLPs; gate, up and down
// matmuls, Appendix C_expert = 6Kdm) and the bf16 router projection.
//
// bf16, many rows: a persistent warp-specialised tcgen05 kernel.
//   warp 0      TMA producer: A tile (128 rows x 64) and B tile (BN rows x 64)
//               per k-block into a STAGES-deep shared-memory ring (128-byte
//               swizzle), completion on mbarriers.
//   warp 1      TMEM allocator and MMA issuer: one thread issues
//               tcgen05.mma.cta_group::1.kind::f16 (M=128, N=BN, K=16) into a
//               double-buffered fp32 accumulator in tensor memory.
//   warps 2..   epilogue (EW warps, 8 by default: two per TMEM lane
//               quarter, each on half of the tile's columns): tcgen05.ld of
//               the accumulator, one row per thread, fused SwiGLU / bf16 /
//               fp32+bias conversion, stores to global.
// Tiles: for every group (expert) g, ceil(rows_g / 128) M-tiles times
// N / BN N-tiles; see tile_coords for the order. Rows past the group's end are
// computed on whatever TMA loaded (zeros past the tensor end) and never
// stored.
// bf16, few rows per expert (decode): the weights-stationary tcgen05 kernel
// k_moe_ws (expert weights as M, the expert's tokens as N).
// f32: CUDA-core kernels (exact fp32 products, fp32 accumulation).
#include <mutex>

#include <cudaTypedefs.h>

#include "decomoe_internal.cuh"

// Kernel choice for the bf16 expert GEMMs: the weights-stationary k_moe_ws
// when the average expert gets at most DECOMOE_WS_MAX_AVG_ROWS rows (decode
// sizes: every tile streams its own weight slice), the tokens-as-M k_gemm_tc
// otherwise (prefill: faster when many rows share an expert's weights).
#ifndef DECOMOE_WS_MAX_AVG_ROWS
#define DECOMOE_WS_MAX_AVG_ROWS 8
#endif

namespace decomoe {

// ------------------------------------------------------------------ TMA maps
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D bf16 tensor [outer, inner] row-major; box = box_outer rows x box_inner
// columns (64 -> 128-byte swizzle, 32 -> 64-byte swizzle), zero fill out of
// bounds.
int make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                          uint32_t box_outer, uint32_t box_inner) {
  auto fn = encode_fn();
  if (fn == nullptr) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return DECOMOE_ERR_CUDA;
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUtensorMapSwizzle sw = box_inner == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                  estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (%d): inner=%llu outer=%llu box=%ux%u", (int)r,
              (unsigned long long)inner, (unsigned long long)outer, box_outer, box_inner);
    return DECOMOE_ERR_CUDA;
  }
  return DECOMOE_OK;
}

// 3-D bf16 tensor, dims[0] innermost (contiguous), byte strides of dims 1 and
// 2, box[0] = 64 elements (128-byte swizzle); zero fill out of bounds.
int make_tmap_bf16_3d(CUtensorMap* m, const void* base, const uint64_t dims[3], const uint64_t strides[2],
                      const uint32_t box[3]) {
  auto fn = encode_fn();
  if (fn == nullptr) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return DECOMOE_ERR_CUDA;
  }
  cuuint64_t d[3] = {dims[0], dims[1], dims[2]};
  cuuint64_t st[2] = {strides[0], strides[1]};
  cuuint32_t bx[3] = {box[0], box[1], box[2]};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), d, st, bx, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled (3-D) failed (%d): dims=%llu x %llu x %llu box=%u x %u x %u", (int)r,
              (unsigned long long)dims[0], (unsigned long long)dims[1], (unsigned long long)dims[2], box[0], box[1],
              box[2]);
    return DECOMOE_ERR_CUDA;
  }
  return DECOMOE_OK;
}

// ------------------------------------------------------------------ tcgen05 GEMM
// EPI_SWIGLU: columns [0, BN/2) gate, [BN/2, BN) up -> bf16 silu(g)*u.
// EPI_BF16: bf16 store. EPI_F32_BIAS: fp32 + bias[col]. EPI_F32_BIAS_T: the
// accumulator is the transpose of the output (A = router rows, B = tokens):
// out[col * ld + row] = acc + bias[row], columns >= n_valid skipped.
enum { EPI_SWIGLU = 0, EPI_BF16 = 1, EPI_F32_BIAS = 2, EPI_F32_BIAS_T = 3 };

struct TcArgs {
  const int32_t* offsets;  // [ngroups + 1] row offsets (device) or null: one group [0, rows)
  int ngroups;
  int rows;
  int n_per_group;  // B rows per group
  int kdim;
  void* out;
  int64_t out_ld;  // elements
  const float* bias;
  int32_t* status;
  uint64_t limit_ns;
  int n_valid;  // EPI_F32_BIAS_T: number of valid output columns (tokens)
  const int32_t* a_rows;  // GA != 0: A row r is row a_rows[r] of the A tensor (rows entries)
  const uint8_t* a_ptr;   // GA == 2: the A tensor itself (rows of kdim bf16)
  int* sched;             // dynamic scheduling: tile counter, zero at launch (null: static round robin)
  int64_t split_stride;   // KS > 1: elements between the k slices' partial outputs
};

// MP = M-tiles per work item. MP = 1: one 128-row A tile per B tile, two
// accumulator buffers (epilogue overlaps the next tile's MMAs). MP = 2: two
// M-tiles of the same group share each B tile (two M=128 MMAs per k-step,
// 2/3 of the shared-memory traffic per MMA), one buffer of two accumulators.
// OCC = resident CTAs per SM. OCC = 2 halves each CTA's shared memory and
// TMEM (one accumulator, no double buffer): two tiles then share an SM, so
// one CTA's weight streaming overlaps the other's tensor-core work.
template <int BN, int STAGES, int BK_, int MP_ = 1, int OCC_ = 1>
struct TcCfg {
  static constexpr int BM = 128, BK = BK_, MP = MP_, OCC = OCC_;
  static constexpr int A_BYTES = BM * BK * 2;  // one M-tile
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = MP * A_BYTES + B_BYTES;
  static constexpr int NBUF = (MP == 1 && OCC == 1) ? 2 : 1;  // accumulator buffers
  static constexpr int TMEM_COLS = NBUF * MP * BN;             // power of two for BN in {128, 256}
  static constexpr int MAXG = DECOMOE_MAX_E;
  static constexpr int TQ = 4;  // depth of the tile-id queue (dynamic scheduling)
  static constexpr int NBARS = 2 * STAGES + 5 + 2 * TQ;
  static constexpr size_t SMEM =
      1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + NBARS * 8 + 2 * (MAXG + 1) * 4 + 16 + TQ * 4;
};

// Work item -> (group, M-tile inside the group, N-tile). M-tiles are visited
// alternately from the two ends of the group-ordered list (first, last,
// second, second-to-last, ...), each with all its N-tiles back to back. With
// experts ordered by routed mass, the front holds large experts whose weight
// tiles are shared by many M-tiles (L2 / tensor bound) and the back small
// experts whose weights stream from HBM once; mixing them in every wave keeps
// both HBM and the tensor pipes busy instead of running the two phases one
// after the other.
__device__ __forceinline__ void tile_coords(int tile, int NT, const int* s_mt, int G, int& grp, int& mt,
                                            int& nb) {
  const int mtot = s_mt[G];
  const int j = tile / NT;
  nb = tile - j * NT;
  const int mtg = (j & 1) ? (mtot - 1 - (j >> 1)) : (j >> 1);
  int lo = 0, hi = G - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_mt[mid] <= mtg)
      lo = mid;
    else
      hi = mid - 1;
  }
  grp = lo;
  mt = mtg - s_mt[lo];
}

// EW epilogue warps (4 or 8): with 8, two warps share each 32-lane TMEM
// quarter and split its column chunks, so the epilogue's latency is hidden.
// GA: how A tiles reach shared memory. 0: tiled TMA of rows [row0, row0+128)
// of A. 2: four extra warps, one A row per thread, 16-byte cp.async of the
// rows a_rows[row0 ..] into the 128-byte-swizzled layout the TMA would
// produce; each thread's copies complete on the stage's full barrier.
// KS: split of the k loop. Work item = (output tile, k slice); slice s runs
// k-blocks [s*KB/KS, (s+1)*KB/KS) and writes its partial sums to
// out + s * split_stride (EPI_F32_BIAS_T only; the caller adds the slices).
template <int BN, int EPI, int STAGES, int BK, int GA = 0, int MP = 1, int EW = 8, int OCC = 1, int KS = 1>
__global__ void __launch_bounds__(64 + 32 * EW + (GA == 2 ? 128 : 0), OCC)
    k_gemm_tc(const __grid_constant__ CUtensorMap tma_a, const __grid_constant__ CUtensorMap tma_b,
              const TcArgs g) {
  using C = TcCfg<BN, STAGES, BK, MP, OCC>;
  static_assert(GA == 0 || GA == 2, "A rows by tiled TMA (0) or by cp.async gather (2)");
  static_assert(!(GA != 0 && MP != 1), "gathered A takes one M-tile per work item");
  static_assert(GA != 2 || BK == 64, "the cp.async gather writes 128-byte swizzled rows");
  static_assert(KS == 1 || (EPI == EPI_F32_BIAS_T && MP == 1 && GA == 0), "k split: transposed fp32 partials only");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sA = raw + pad;
  const uint32_t sB = sA + STAGES * MP * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
  int* s_off = reinterpret_cast<int*>(bars + C::NBARS);
  int* s_mt = s_off + (C::MAXG + 1);
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(s_mt + (C::MAXG + 1));
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  volatile int* s_tq = reinterpret_cast<volatile int*>(s_tmem + 4);  // [TQ] tile ids

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t bar0 = smem_u32(bars);
  // barrier slots: full[STAGES] | empty[STAGES] | tfull[2] | tempty[2] | drain | tqfull[TQ] | tqempty[TQ]
#define FULL_BAR(s) (bar0 + 8u * (s))
#define EMPTY_BAR(s) (bar0 + 8u * (STAGES + (s)))
#define TFULL_BAR(a) (bar0 + 8u * (2 * STAGES + (a)))
#define TEMPTY_BAR(a) (bar0 + 8u * (2 * STAGES + 2 + (a)))
#define DRAIN_BAR (bar0 + 8u * (2 * STAGES + 4))
#define TQF_BAR(i) (bar0 + 8u * (2 * STAGES + 5 + (i)))
#define TQE_BAR(i) (bar0 + 8u * (2 * STAGES + 5 + C::TQ + (i)))

  const int G = g.ngroups;
  if (threadIdx.x == 0) {
    *s_abort = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(FULL_BAR(s), GA == 2 ? 1 + 128 : 1);  // + one arrival per cp.async A-row thread
      mbar_init(EMPTY_BAR(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(TFULL_BAR(a), 1);
      mbar_init(TEMPTY_BAR(a), 32 * EW);
    }
    mbar_init(DRAIN_BAR, 1);
    for (int i = 0; i < C::TQ; ++i) {
      mbar_init(TQF_BAR(i), 1);
      mbar_init(TQE_BAR(i), 1 + EW);  // the MMA thread and lane 0 of every epilogue warp
    }
    fence_mbar_init();
  }
  // wait for the earlier kernels' results; the next kernel is released only
  // at the end (its CTAs would otherwise sit resident through this one)
  pdl_wait();
  for (int i = threadIdx.x; i <= G; i += blockDim.x)
    s_off[i] = (g.offsets != nullptr) ? g.offsets[i] : (i == 0 ? 0 : g.rows);
  __syncthreads();
  if (warp == 2) {
    // exclusive scan of work units (MP M-tiles) per group: s_mt[g] = first unit of g
    const int per = (G + 31) / 32;  // <= 8
    int loc[8];
    int sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      loc[i] = 0;
      const int gi = lane * per + i;
      if (i < per && gi < G) {
        const int n = s_off[gi + 1] - s_off[gi];
        loc[i] = n > 0 ? (n + C::BM * MP - 1) / (C::BM * MP) : 0;
      }
      sum += loc[i];
    }
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    int run = incl - sum;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int gi = lane * per + i;
      if (i < per && gi < G) s_mt[gi] = run;
      run += loc[i];
    }
    if (lane == 31) s_mt[G] = incl;
  }
  __syncthreads();
  const int NT = g.n_per_group / BN;
  const int total = s_mt[G] * NT * KS;
  if (static_cast<int>(blockIdx.x) >= total) return;  // before any TMEM or TMA use

  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<uint32_t*>(s_tmem)), C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  const int KB = g.kdim / C::BK / KS;  // k-blocks per work item

  // Tile sequence of this CTA. Static: blockIdx.x, + gridDim.x, ... Dynamic:
  // the producer takes the next id from the global counter and passes it to
  // the MMA and epilogue warps through a TQ-deep shared-memory queue; -1 ends.
  const bool dyn = GA == 0 && g.sched != nullptr;
  auto static_tile = [&](int i) -> int {
    const int t = static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x);
    return t < total ? t : -1;
  };
  auto produce_tile = [&](int i) -> int {  // producer thread; returns -2 on timeout
    if (!dyn) return static_tile(i);
    const int slot = i % C::TQ;
    const uint32_t qph = (i / C::TQ) & 1;
    if (!mbar_wait(TQE_BAR(slot), qph ^ 1u, g.limit_ns, s_abort)) return -2;
    int t = atomicAdd(g.sched, 1);
    if (t >= total) t = -1;
    s_tq[slot] = t;
    mbar_arrive(TQF_BAR(slot));
    return t;
  };
  auto consume_tile = [&](int i, bool arrive) -> int {  // returns -2 on timeout
    if (!dyn) return static_tile(i);
    const int slot = i % C::TQ;
    const uint32_t qph = (i / C::TQ) & 1;
    if (!mbar_wait(TQF_BAR(slot), qph, g.limit_ns, s_abort)) return -2;
    const int t = s_tq[slot];
    if (arrive) mbar_arrive(TQE_BAR(slot));
    return t;
  };

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0 issues)
    if (lane == 0) {
      tma_prefetch_desc(&tma_a);
      tma_prefetch_desc(&tma_b);
    }
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    uint32_t armed = 0;  // bit s: stage s was ever filled
    uint32_t armed_ph = 0;
    for (int ti = 0;; ++ti) {
      int tile = 0;
      if (lane == 0) tile = produce_tile(ti);
      tile = __shfl_sync(0xffffffffu, tile, 0);
      if (tile == -2) {
        ok = false;
        break;
      }
      if (tile < 0) break;
      int grp, mt, nb;
      tile_coords(tile / KS, NT, s_mt, G, grp, mt, nb);
      const int row0 = s_off[grp] + mt * MP * C::BM;
      const int brow = grp * g.n_per_group + nb * BN;
      const int kbase = (tile % KS) * KB;  // first k-block of this work item's slice
      const bool has2 = MP == 2 && row0 + C::BM < s_off[grp + 1];  // second M-tile has rows
      if (lane == 0) {
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(FULL_BAR(stage), (GA == 2 ? 0 : (has2 ? 2 : 1) * C::A_BYTES) + C::B_BYTES);
          if constexpr (GA == 0) {
            tma_load_2d(sA + stage * MP * C::A_BYTES, &tma_a, FULL_BAR(stage), (kbase + kb) * C::BK, row0);
            if (has2)
              tma_load_2d(sA + (stage * MP + 1) * C::A_BYTES, &tma_a, FULL_BAR(stage), (kbase + kb) * C::BK,
                          row0 + C::BM);
          }
          tma_load_2d(sB + stage * C::B_BYTES, &tma_b, FULL_BAR(stage), (kbase + kb) * C::BK, brow);
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
    }
    if (lane == 0 && !ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      // let every copy this thread started land before the CTA can exit
      int no_abort = 0;
      for (int s = 0; s < STAGES; ++s)
        if ((armed >> s) & 1u) mbar_wait(FULL_BAR(s), (armed_ph >> s) & 1u, g.limit_ns, &no_abort);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------ MMA issuer
    constexpr uint32_t IDESC = idesc_bf16_f32(C::BM, BN);
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true, issued = false;
    for (int it = 0;; ++it) {
      const int tile = consume_tile(it, true);
      if (tile == -2) {
        ok = false;
        break;
      }
      if (tile < 0) break;
      const int acc = it % C::NBUF;
      const uint32_t aph = (it / C::NBUF) & 1;
      bool has2 = false;
      if constexpr (MP == 2) {
        int grp, mt, nb;
        tile_coords(tile / KS, NT, s_mt, G, grp, mt, nb);
        has2 = s_off[grp] + (mt * 2 + 1) * C::BM < s_off[grp + 1];
      }
      if (!mbar_wait(TEMPTY_BAR(acc), aph ^ 1u, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t dt = tmem_base + static_cast<uint32_t>(acc * BN);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(FULL_BAR(stage), ph, g.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if constexpr (GA == 2) fence_proxy_async_smem();  // A rows came through the generic proxy
        const uint64_t ad = smem_desc_kmajor<BK>(sA + stage * MP * C::A_BYTES);
        const uint64_t bd = smem_desc_kmajor<BK>(sB + stage * C::B_BYTES);
#pragma unroll
        for (int kk = 0; kk < C::BK / 16; ++kk) {
          tc_mma_f16(dt, ad + 2u * kk, bd + 2u * kk, IDESC, (kb | kk) != 0 ? 1u : 0u);
          if (MP == 2 && has2)
            tc_mma_f16(tmem_base + BN, ad + static_cast<uint64_t>(C::A_BYTES >> 4) + 2u * kk, bd + 2u * kk, IDESC,
                       (kb | kk) != 0 ? 1u : 0u);
        }
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
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      if (issued) {
        int no_abort = 0;
        tc_commit(DRAIN_BAR);
        mbar_wait(DRAIN_BAR, 0, g.limit_ns, &no_abort);
      }
    }
  } else if (GA == 2 && warp >= 2 + EW) {
    // ------------------------------------------------ A rows by cp.async:
    // the 128 threads copy the tile's 128 A rows (token rows a_rows[row0 +
    // i] of the A tensor), 8 x 16 bytes per row per k-block, eight lanes per
    // row so each warp instruction reads four whole 128-byte row segments.
    // Chunk c of tile row i lands at i*128 + ((c ^ (i & 7)) * 16): the
    // 128-byte-swizzled layout the TMA would write.
    const int t = threadIdx.x - 32 * (2 + EW);
    const int c = lane & 7;                      // 16-byte chunk of the row
    const int i0 = (t >> 5) * 32 + (lane >> 3);  // rows i0 + 4j, j < 8
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    for (int ti = 0;; ++ti) {
      const int tile = static_tile(ti);
      if (tile < 0) break;
      int grp, mt, nb;
      tile_coords(tile / KS, NT, s_mt, G, grp, mt, nb);
      const int row0 = s_off[grp] + mt * C::BM;
      const uint8_t* src[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int r = row0 + i0 + 4 * j;
        const int src_row = (r < g.rows) ? g.a_rows[r] : 0;  // rows past the end: any valid row, never stored
        src[j] = g.a_ptr + static_cast<int64_t>(src_row) * g.kdim * 2 + c * 16;
      }
      for (int kb = 0; kb < KB; ++kb) {
        bool got = true;
        if (lane == 0) got = mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort);
        got = __shfl_sync(0xffffffffu, got, 0);
        if (!got) {
          ok = false;
          break;
        }
        const uint32_t dst = sA + stage * C::A_BYTES;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int i = i0 + 4 * j;
          cp_async16(dst + static_cast<uint32_t>(i) * 128u + (static_cast<uint32_t>(c ^ (i & 7)) << 4),
                     src[j] + kb * (C::BK * 2));
        }
        cp_async_mbar_arrive_noinc(FULL_BAR(stage));
        if (++stage == STAGES) {
          stage = 0;
          ph ^= 1u;
        }
      }
      if (!ok) break;
    }
    cp_async_wait_all();  // every copy lands before the CTA can exit
    if (!ok && lane == 0) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
    }
  } else if (warp >= 2) {
    // ------------------------------------------------ epilogue
    const int q = warp & 3;            // TMEM lanes [32q, 32q + 32) belong to this warp
    const int wp = (warp - 2) >> 2;    // which of the quarter's warps (0 .. EW/4 - 1)
    constexpr int WPQ = EW / 4;        // warps per quarter: column chunks are dealt round robin
    bool ok = true;
    for (int it = 0;; ++it) {
      int tile = 0;
      if (lane == 0) tile = consume_tile(it, true);
      tile = __shfl_sync(0xffffffffu, tile, 0);
      if (tile == -2) {
        ok = false;
        break;
      }
      if (tile < 0) break;
      const int acc = it % C::NBUF;
      const uint32_t aph = (it / C::NBUF) & 1;
      int grp, mt, nb;
      tile_coords(tile / KS, NT, s_mt, G, grp, mt, nb);
      const int row_end = s_off[grp + 1];
      if (!mbar_wait(TFULL_BAR(acc), aph, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
#pragma unroll 1
      for (int sub = 0; sub < MP; ++sub) {
      const int row0 = s_off[grp] + (mt * MP + sub) * C::BM;
      if (sub > 0 && row0 >= row_end) break;  // no second M-tile in this unit
      const int grow = row0 + q * 32 + lane;
      const bool valid = grow < row_end;
      const uint32_t tb =
          tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>((acc + sub) * BN);
      if constexpr (EPI == EPI_SWIGLU) {
        // columns hold blocks of GU gate then GU up columns of the same
        // features: features nb*BN/2 + half*GU + c
        constexpr int GU = DECOMOE_GU_BLOCK;
        static_assert(BN % (2 * GU) == 0, "N tile must hold whole gate/up blocks");
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(g.out);
#pragma unroll 1
        for (int cc = 32 * wp; cc < BN / 2; cc += 32 * WPQ) {
          const int half = cc / GU, c = cc % GU;
          uint32_t gr[32], ur[32];
          tmem_ld32(tb + half * 2 * GU + c, gr);
          tmem_ld32(tb + half * 2 * GU + GU + c, ur);
          tc_wait_ld();
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float g0 = __uint_as_float(gr[2 * i]), g1 = __uint_as_float(gr[2 * i + 1]);
            const float u0 = __uint_as_float(ur[2 * i]), u1 = __uint_as_float(ur[2 * i + 1]);
            pk[i] = pack_bf16x2(silu_f(g0) * u0, silu_f(g1) * u1);
          }
          if (valid) {
            uint4* dst = reinterpret_cast<uint4*>(out + static_cast<int64_t>(grow) * g.out_ld +
                                                  nb * (BN / 2) + cc);
#pragma unroll
            for (int v = 0; v < 4; ++v)
              dst[v] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
          }
        }
      } else if constexpr (EPI == EPI_BF16) {
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(g.out);
#pragma unroll 1
        for (int c = 32 * wp; c < BN; c += 32 * WPQ) {
          uint32_t r[32];
          tmem_ld32(tb + c, r);
          tc_wait_ld();
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 16; ++i)
            pk[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
          if (valid) {
            uint4* dst =
                reinterpret_cast<uint4*>(out + static_cast<int64_t>(grow) * g.out_ld + nb * BN + c);
#pragma unroll
            for (int v = 0; v < 4; ++v)
              dst[v] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
          }
        }
      } else if constexpr (EPI == EPI_F32_BIAS_T) {
        // row = router row (expert), columns = tokens nb*BN + c; with a k
        // split, slice (tile % KS) writes its partial sums without the bias
        float* out = static_cast<float*>(g.out) + static_cast<int64_t>(tile % KS) * g.split_stride;
        const float bv = (KS == 1 && valid && g.bias) ? g.bias[grow] : 0.f;
        const int n0 = nb * BN;
        if constexpr (BN == 16) {
          if (wp == 0) {
          uint32_t r[16];
          tmem_ld16(tb, r);
          tc_wait_ld();
          if (valid) {
#pragma unroll
            for (int c = 0; c < 16; ++c)
              if (n0 + c < g.n_valid) out[static_cast<int64_t>(n0 + c) * g.out_ld + grow] = __uint_as_float(r[c]) + bv;
          }
          }
        } else {
#pragma unroll 1
          for (int c0 = 32 * wp; c0 < BN; c0 += 32 * WPQ) {
            uint32_t r[32];
            tmem_ld32(tb + c0, r);
            tc_wait_ld();
            if (valid) {
#pragma unroll
              for (int c = 0; c < 32; ++c)
                if (n0 + c0 + c < g.n_valid)
                  out[static_cast<int64_t>(n0 + c0 + c) * g.out_ld + grow] = __uint_as_float(r[c]) + bv;
            }
          }
        }
      } else {
        float* out = static_cast<float*>(g.out);
#pragma unroll 1
        for (int c = 32 * wp; c < BN; c += 32 * WPQ) {
          uint32_t r[32];
          tmem_ld32(tb + c, r);
          tc_wait_ld();
          if (valid) {
            float4* dst =
                reinterpret_cast<float4*>(out + static_cast<int64_t>(grow) * g.out_ld + nb * BN + c);
            const float* bptr = g.bias ? g.bias + nb * BN + c : nullptr;
#pragma unroll
            for (int v = 0; v < 8; ++v) {
              float4 o;
              o.x = __uint_as_float(r[4 * v + 0]) + (bptr ? bptr[4 * v + 0] : 0.f);
              o.y = __uint_as_float(r[4 * v + 1]) + (bptr ? bptr[4 * v + 1] : 0.f);
              o.z = __uint_as_float(r[4 * v + 2]) + (bptr ? bptr[4 * v + 2] : 0.f);
              o.w = __uint_as_float(r[4 * v + 3]) + (bptr ? bptr[4 * v + 3] : 0.f);
              dst[v] = o;
            }
          }
        }
      }
      }  // sub
      tc_fence_before();
      mbar_arrive(TEMPTY_BAR(acc));
    }
    if (!ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
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
#undef TQF_BAR
#undef TQE_BAR
}

// A: [rows, kdim], or with GA == 2 the source tensor [a_tensor_rows, kdim]
// whose row a_rows[r] is A row r.
template <int BN, int EPI, int STAGES, int BK, int GA = 0, int MP = 1, int EW = 8, int OCC = 1, int KS = 1>
static int launch_tc(const void* A, int rows, int kdim, const void* B, int64_t b_rows,
                     const int32_t* offsets, int ngroups, int n_per_group, void* out,
                     int64_t out_ld, const float* bias, int32_t* status, cudaStream_t s, int n_valid = 0,
                     const int32_t* a_rows = nullptr, int64_t a_tensor_rows = 0, int* sched = nullptr,
                     int64_t split_stride = 0) {
  using C = TcCfg<BN, STAGES, BK, MP, OCC>;
  CUtensorMap ta, tb;
  if (GA == 2)
    ta = CUtensorMap{};  // A is read with cp.async, not TMA
  else
    DM_RET(make_tmap_bf16(&ta, A, static_cast<uint64_t>(kdim), static_cast<uint64_t>(rows), C::BM, BK));
  DM_RET(make_tmap_bf16(&tb, B, static_cast<uint64_t>(kdim), static_cast<uint64_t>(b_rows), BN, BK));
  TcArgs g;
  g.offsets = offsets;
  g.ngroups = ngroups;
  g.rows = rows;
  g.n_per_group = n_per_group;
  g.kdim = kdim;
  g.out = out;
  g.out_ld = out_ld;
  g.bias = bias;
  g.status = status;
  g.limit_ns = static_cast<uint64_t>(wait_limit_ns());
  g.n_valid = n_valid;
  g.a_rows = a_rows;
  g.a_ptr = static_cast<const uint8_t*>(A);
  g.sched = sched;
  g.split_stride = split_stride;
  if (sched != nullptr) DM_CUDA_CHECK(cudaMemsetAsync(sched, 0, sizeof(int), s));
  auto kern = k_gemm_tc<BN, EPI, STAGES, BK, GA, MP, EW, OCC, KS>;
  static_assert(C::SMEM <= 232448, "shared memory budget");
  DM_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(C::SMEM)));
  const int64_t ub_tiles =
      (static_cast<int64_t>(rows) / C::BM + ngroups) * static_cast<int64_t>(n_per_group / BN) * KS;
  const int64_t cap = static_cast<int64_t>(sm_count()) * OCC;
  const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(cap, ub_tiles)));
  DM_CUDA_CHECK(launch_pdl(kern, dim3(grid), dim3(64 + 32 * EW + (GA == 2 ? 128 : 0)), C::SMEM, s, ta, tb, g));
  return DECOMOE_OK;
}

// ------------------------------------------------------------------ weights-stationary grouped GEMM
// D[w, t] = sum_k W[e][wrow0 + w, k] * X[row0 + t, k]: the expert's weight rows
// are the M operand (128 per tile, always full) and its tokens the N operand
// (up to 256 per tile, MMA width rounded up to 16). No M padding, so a ragged,
// skewed expert population costs only what it routes; small experts (and the
// decode sizes) become pure weight streaming with every tile reading its own
// 128-row weight slice once. Roles as in k_gemm_tc (TMA warp, MMA warp, four
// epilogue warps, double-buffered 256-column TMEM accumulators).
//
// Tiles: per expert e, (wrows / 128) weight blocks x ceil(n_e / 256) token
// chunks, chunk innermost (consecutive tiles share a weight block, so it is
// read from HBM once and from L2 after); the global list is visited
// alternately from both ends, as in k_gemm_tc.
//
// SwiGLU epilogue: with the 64-row gate/up interleave a weight block holds 64
// gate rows (TMEM lanes 0..63) and the 64 up rows of the same features (lanes
// 64..127). The warps owning lanes 64..127 pass their up values through a
// small double-buffered shared-memory exchange to the warps owning the gate
// lanes of the same features, which write h.
struct WsArgs {
  const int32_t* offsets;  // [G + 1] token row offsets per expert
  int G;                   // experts [0, G)
  int rows;                // token rows of the activation tensor
  int wrows;               // weight rows per expert (2m gate/up, d down)
  int kdim;
  void* out;
  int64_t out_ld;
  int32_t* status;
  uint64_t limit_ns;
  const int32_t* b_rows;  // GATHER_B: token row r is row b_rows[r] of the activation tensor
};

#ifndef DECOMOE_WS_BOX
#define DECOMOE_WS_BOX 32
#endif
constexpr int WS_BM = 128, WS_BK = 64, WS_BOX = DECOMOE_WS_BOX;

// BN: token chunk (the MMA's N), one chunk per (expert, weight block) tile
// when an expert has at most BN rows; smaller chunks leave shared memory for
// a deeper weight-streaming ring.
template <int STAGES, bool SWIGLU, int BN = 256>
struct WsCfg {
  static constexpr int WS_BN = BN;
  static constexpr int A_BYTES = WS_BM * WS_BK * 2;
  static constexpr int B_BYTES = WS_BN * WS_BK * 2;
  static constexpr int BOX_BYTES = WS_BOX * WS_BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * WS_BN;
  static constexpr int MAXG = DECOMOE_MAX_E;
  static constexpr int NBARS = 2 * STAGES + 5;
  static constexpr int XCH_BYTES = SWIGLU ? 2 * 2 * 32 * 32 * 4 : 0;  // up values, double-buffered
  static constexpr int OUT_COLS = SWIGLU ? WS_BM / 2 : WS_BM;            // output features per tile
  static constexpr int STILE_BYTES = 2 * 32 * OUT_COLS * 2;              // [2][32 tokens][OUT_COLS] bf16
  static constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + XCH_BYTES + STILE_BYTES +
                                 NBARS * 8 + 2 * (MAXG + 1) * 4 + 16;
};

// Most stages of a WsCfg<., SWIGLU, BN> that fit the shared-memory budget.
template <bool SWIGLU, int BN>
constexpr int ws_max_stages() {
  constexpr size_t fixed = WsCfg<1, SWIGLU, BN>::SMEM - WsCfg<1, SWIGLU, BN>::STAGE_BYTES - 2 * 8;
  constexpr size_t per = WsCfg<1, SWIGLU, BN>::STAGE_BYTES + 2 * 8;
  constexpr int n = static_cast<int>((232448 - fixed) / per);
  return n > 12 ? 12 : n;
}

struct WsTile {
  int g, wb, row0, ntok;
};

template <int WS_BN>
__device__ __forceinline__ WsTile ws_tile(int t, int total, const int* s_tt, const int* s_off, int G, int nwb) {
  const int tp = (t & 1) ? (total - 1 - (t >> 1)) : (t >> 1);
  int lo = 0, hi = G - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_tt[mid] <= tp)
      lo = mid;
    else
      hi = mid - 1;
  }
  WsTile r;
  r.g = lo;
  const int n = s_off[lo + 1] - s_off[lo];
  const int nch = (n + WS_BN - 1) / WS_BN;
  const int local = tp - s_tt[lo];
  r.wb = local / nch;
  const int c = local - r.wb * nch;
  r.row0 = s_off[lo] + c * WS_BN;
  r.ntok = min(WS_BN, n - c * WS_BN);
  return r;
}


template <bool SWIGLU, int STAGES, bool GATHER_B = false, int BN = 256>
__global__ void __launch_bounds__(192, 1)
    k_moe_ws(const __grid_constant__ CUtensorMap tma_w, const __grid_constant__ CUtensorMap tma_x,
             const WsArgs g) {
  using C = WsCfg<STAGES, SWIGLU, BN>;
  constexpr int WS_BN = BN;
  __shared__ int s_brow[GATHER_B ? WS_BN : 1];
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sA = raw + pad;
  const uint32_t sB = sA + STAGES * C::A_BYTES;
  float* xch = reinterpret_cast<float*>(smem + STAGES * C::STAGE_BYTES);
  __nv_bfloat16* stile = reinterpret_cast<__nv_bfloat16*>(smem + STAGES * C::STAGE_BYTES + C::XCH_BYTES);
  uint64_t* bars =
      reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES + C::XCH_BYTES + C::STILE_BYTES);
  int* s_off = reinterpret_cast<int*>(bars + C::NBARS);
  int* s_tt = s_off + (C::MAXG + 1);
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(s_tt + (C::MAXG + 1));
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t bar0 = smem_u32(bars);
#define FULL_BAR(s) (bar0 + 8u * (s))
#define EMPTY_BAR(s) (bar0 + 8u * (STAGES + (s)))
#define TFULL_BAR(a) (bar0 + 8u * (2 * STAGES + (a)))
#define TEMPTY_BAR(a) (bar0 + 8u * (2 * STAGES + 2 + (a)))
#define DRAIN_BAR (bar0 + 8u * (2 * STAGES + 4))

  const int G = g.G;
  const int nwb = g.wrows / WS_BM;
  if (threadIdx.x == 0) {
    *s_abort = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(FULL_BAR(s), 1);
      mbar_init(EMPTY_BAR(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(TFULL_BAR(a), 1);
      mbar_init(TEMPTY_BAR(a), 128);
    }
    mbar_init(DRAIN_BAR, 1);
    fence_mbar_init();
  }
  // wait for the earlier kernels' results; the next kernel is released only
  // at the end (its CTAs would otherwise sit resident through this one)
  pdl_wait();
  for (int i = threadIdx.x; i <= G; i += blockDim.x) s_off[i] = g.offsets[i];
  __syncthreads();
  if (warp == 2) {
    // s_tt[e] = first tile of expert e = sum over earlier experts of nwb * chunks
    const int per = (G + 31) / 32;
    int loc[8];
    int sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      loc[i] = 0;
      const int gi = lane * per + i;
      if (i < per && gi < G) {
        const int n = s_off[gi + 1] - s_off[gi];
        loc[i] = n > 0 ? ((n + WS_BN - 1) / WS_BN) * nwb : 0;
      }
      sum += loc[i];
    }
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    int run = incl - sum;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int gi = lane * per + i;
      if (i < per && gi < G) s_tt[gi] = run;
      run += loc[i];
    }
    if (lane == 31) s_tt[G] = incl;
  }
  __syncthreads();
  const int total = s_tt[G];
  if (static_cast<int>(blockIdx.x) >= total) return;

  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<uint32_t*>(s_tmem)), C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  const int KB = g.kdim / WS_BK;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0
    // issues; with GATHER_B the warp first reads the tile's token row indices)
    if (lane == 0) {
      tma_prefetch_desc(&tma_w);
      tma_prefetch_desc(&tma_x);
    }
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    uint32_t armed = 0, armed_ph = 0;
    // an expert of one token chunk reads each weight block once: evict-first
    // in L2 (blocks of larger experts are re-read by their next chunks)
    const uint64_t pol_once = policy_evict_first();
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      const WsTile T = ws_tile<WS_BN>(t, total, s_tt, s_off, G, nwb);
      const int wrow0 = T.g * g.wrows + T.wb * WS_BM;
      const bool once = s_off[T.g + 1] - s_off[T.g] <= WS_BN;
      int nload;       // TMA copies for B per k-block
      uint32_t bytes;  // bytes landing per stage
      if constexpr (GATHER_B) {
        for (int i = lane; i < WS_BN; i += 32)
          s_brow[i] = (i < T.ntok) ? g.b_rows[T.row0 + i] : 0;  // padding rows: any valid row, never stored
        __syncwarp();
        nload = (T.ntok + 3) / 4;
        bytes = C::A_BYTES + nload * 4 * WS_BK * 2;
      } else {
        nload = (T.ntok + WS_BOX - 1) / WS_BOX;
        bytes = C::A_BYTES + nload * C::BOX_BYTES;
      }
      if (lane == 0) {
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(FULL_BAR(stage), bytes);
          if (once)
            tma_load_2d_hint(sA + stage * C::A_BYTES, &tma_w, FULL_BAR(stage), kb * WS_BK, wrow0, pol_once);
          else
            tma_load_2d(sA + stage * C::A_BYTES, &tma_w, FULL_BAR(stage), kb * WS_BK, wrow0);
          const uint32_t dB = sB + stage * C::B_BYTES;
          if constexpr (GATHER_B) {
            for (int i = 0; i < nload; ++i)
              tma_gather4(dB + i * 4 * WS_BK * 2, &tma_x, FULL_BAR(stage), kb * WS_BK, s_brow[4 * i],
                          s_brow[4 * i + 1], s_brow[4 * i + 2], s_brow[4 * i + 3]);
          } else {
            for (int i = 0; i < nload; ++i)
              tma_load_2d(dB + i * C::BOX_BYTES, &tma_x, FULL_BAR(stage), kb * WS_BK, T.row0 + i * WS_BOX);
          }
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
    }
    if (lane == 0 && !ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      int no_abort = 0;
      for (int s = 0; s < STAGES; ++s)
        if ((armed >> s) & 1u) mbar_wait(FULL_BAR(s), (armed_ph >> s) & 1u, g.limit_ns, &no_abort);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------ MMA issuer
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true, issued = false;
    int it = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
      const WsTile T = ws_tile<WS_BN>(t, total, s_tt, s_off, G, nwb);
      const uint32_t idesc = idesc_bf16_f32(WS_BM, (T.ntok + 15) & ~15);
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait(TEMPTY_BAR(acc), aph ^ 1u, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t dt = tmem_base + static_cast<uint32_t>(acc * WS_BN);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(FULL_BAR(stage), ph, g.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = smem_desc_kmajor<WS_BK>(sA + stage * C::A_BYTES);
        const uint64_t bd = smem_desc_kmajor<WS_BK>(sB + stage * C::B_BYTES);
#pragma unroll
        for (int kk = 0; kk < WS_BK / 16; ++kk)
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
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      if (issued) {
        int no_abort = 0;
        tc_commit(DRAIN_BAR);
        mbar_wait(DRAIN_BAR, 0, g.limit_ns, &no_abort);
      }
    }
  } else if (warp >= 2) {
    // ------------------------------------------------ epilogue
    const int q = warp & 3;  // TMEM lanes [32q, 32q + 32)
    __nv_bfloat16* out = static_cast<__nv_bfloat16*>(g.out);
    int it = 0;
    int xpar = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
      const WsTile T = ws_tile<WS_BN>(t, total, s_tt, s_off, G, nwb);
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait(TFULL_BAR(acc), aph, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t tb =
          tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * WS_BN);
      // Each 32-token chunk: accumulator columns -> registers -> (SwiGLU) ->
      // bf16 tile [32 tokens][OUT_COLS features] in shared memory -> 16-byte
      // row stores to out[token, feature]. Two named barriers per chunk over
      // the four epilogue warps; the exchange and tile buffers alternate.
      constexpr int OC = C::OUT_COLS;
      const int et = threadIdx.x - 64;  // 0..127 among the epilogue warps
      const int fbase = T.wb * OC;      // first output feature of this tile
#pragma unroll 1
      for (int c0 = 0; c0 < T.ntok; c0 += 32) {
        uint32_t r[32];
        tmem_ld32(tb + c0, r);
        tc_wait_ld();
        __nv_bfloat16* st = stile + xpar * (32 * OC);
        if constexpr (SWIGLU) {
          const bool is_gate = q < 2;
          const int pr = q & 1;
          float* xb = xch + (xpar * 2 + pr) * 1024;  // [32 columns][32 lanes]
          if (!is_gate) {
#pragma unroll
            for (int c = 0; c < 32; ++c) xb[c * 32 + lane] = __uint_as_float(r[c]);
          }
          named_bar_sync(1, 128);
          if (is_gate) {
#pragma unroll
            for (int c = 0; c < 32; ++c)
              st[c * OC + pr * 32 + lane] = __float2bfloat16_rn(silu_f(__uint_as_float(r[c])) * xb[c * 32 + lane]);
          }
        } else {
#pragma unroll
          for (int c = 0; c < 32; ++c) st[c * OC + q * 32 + lane] = __float2bfloat16_rn(__uint_as_float(r[c]));
        }
        named_bar_sync(1, 128);
        const int nc = min(32, T.ntok - c0);
        constexpr int VPR = OC / 8;  // 16-byte vectors per token row
#pragma unroll
        for (int v = et; v < 32 * VPR; v += 128) {
          const int row = v / VPR, cv = v - row * VPR;
          if (row < nc) {
            const uint4 val = *reinterpret_cast<const uint4*>(st + row * OC + cv * 8);
            *reinterpret_cast<uint4*>(out + static_cast<int64_t>(T.row0 + c0 + row) * g.out_ld + fbase + cv * 8) = val;
          }
        }
        xpar ^= 1;
      }
      tc_fence_before();
      mbar_arrive(TEMPTY_BAR(acc));
    }
    if (!ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
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
}

// ------------------------------------------------------------------ fused decode FFN
// Gate/up and down of the weights-stationary decode path in one persistent
// launch. Work items: every gate/up tile of k_moe_ws<true> first, then every
// down tile of k_moe_ws<false> (each list in k_moe_ws's order), handed out
// round robin. A down tile of expert e reads h rows that the gate/up tiles
// of e write, so after storing its h slice a gate/up tile bumps ready[e]
// (release), and a down tile first issues the loads of its own weight
// k-blocks (they depend on nothing), then waits until ready[e] counts all of
// e's gate/up tiles (acquire, bounded) before loading its h rows. CTAs whose
// first item is a down tile thus stream their weights while the gate/up
// tiles run, and no launch separates the two GEMMs. Deadlock-free with at
// most one CTA per SM and grid <= SMs: gate/up items never wait, and every
// CTA reaches its gate/up items before any down item. ready[] must be zero at
// launch (the layer's routing launch clears it).
struct WsFfnArgs {
  const int32_t* offsets;  // [G + 1] token row offsets per expert
  int G;
  int rows;
  int wrows1, kdim1;  // gate/up: 2m weight rows per expert, K = d
  int wrows2, kdim2;  // down: d weight rows per expert, K = m
  void* h;            // [rows, m] bf16, gate/up output and down input
  int64_t h_ld;
  void* y;  // [rows, d] bf16
  int64_t y_ld;
  int32_t* ready;  // [G] finished gate/up tiles per expert; zero at launch
  int32_t* status;
  uint64_t limit_ns;
};

template <int STAGES, int BN>
struct WsFfnCfg {
  static constexpr int A_BYTES = WS_BM * WS_BK * 2;
  static constexpr int B_BYTES = BN * WS_BK * 2;
  static constexpr int BOX_BYTES = WS_BOX * WS_BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;
  static constexpr int MAXG = DECOMOE_MAX_E;
  static constexpr int NBARS = 2 * STAGES + 5;
  static constexpr int XCH_BYTES = 2 * 2 * 32 * 32 * 4;   // SwiGLU up values, double-buffered
  static constexpr int STILE_BYTES = 2 * 32 * WS_BM * 2;  // [2][32 tokens][128 features] bf16
  static constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + XCH_BYTES + STILE_BYTES +
                                 NBARS * 8 + 3 * (MAXG + 1) * 4 + 16;
};

template <int BN>
constexpr int ffn_ws_max_stages() {
  constexpr size_t fixed = WsFfnCfg<1, BN>::SMEM - WsFfnCfg<1, BN>::STAGE_BYTES - 2 * 8;
  constexpr size_t per = WsFfnCfg<1, BN>::STAGE_BYTES + 2 * 8;
  constexpr int n = static_cast<int>((232448 - fixed) / per);
  return n > 12 ? 12 : n;
}


template <int STAGES, int BN>
__global__ void __launch_bounds__(192, 1)
    k_ffn_ws(const __grid_constant__ CUtensorMap tma_w1, const __grid_constant__ CUtensorMap tma_x1,
             const __grid_constant__ CUtensorMap tma_w2, const __grid_constant__ CUtensorMap tma_x2,
             const WsFfnArgs g) {
  using C = WsFfnCfg<STAGES, BN>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sA = raw + pad;
  const uint32_t sB = sA + STAGES * C::A_BYTES;
  float* xch = reinterpret_cast<float*>(smem + STAGES * C::STAGE_BYTES);
  __nv_bfloat16* stile = reinterpret_cast<__nv_bfloat16*>(smem + STAGES * C::STAGE_BYTES + C::XCH_BYTES);
  uint64_t* bars =
      reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES + C::XCH_BYTES + C::STILE_BYTES);
  int* s_off = reinterpret_cast<int*>(bars + C::NBARS);
  int* s_tt1 = s_off + (C::MAXG + 1);
  int* s_tt2 = s_tt1 + (C::MAXG + 1);
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(s_tt2 + (C::MAXG + 1));
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t bar0 = smem_u32(bars);
#define FULL_BAR(s) (bar0 + 8u * (s))
#define EMPTY_BAR(s) (bar0 + 8u * (STAGES + (s)))
#define TFULL_BAR(a) (bar0 + 8u * (2 * STAGES + (a)))
#define TEMPTY_BAR(a) (bar0 + 8u * (2 * STAGES + 2 + (a)))
#define DRAIN_BAR (bar0 + 8u * (2 * STAGES + 4))

  const int G = g.G;
  const int nwb1 = g.wrows1 / WS_BM, nwb2 = g.wrows2 / WS_BM;
  if (threadIdx.x == 0) {
    *s_abort = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(FULL_BAR(s), 1);
      mbar_init(EMPTY_BAR(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(TFULL_BAR(a), 1);
      mbar_init(TEMPTY_BAR(a), 128);
    }
    mbar_init(DRAIN_BAR, 1);
    fence_mbar_init();
  }
  pdl_wait();
  for (int i = threadIdx.x; i <= G; i += blockDim.x) s_off[i] = g.offsets[i];
  __syncthreads();
  if (warp == 2 || warp == 3) {
    // s_tt1 / s_tt2[e] = first gate/up / down item of expert e
    const int nwb = warp == 2 ? nwb1 : nwb2;
    int* s_tt = warp == 2 ? s_tt1 : s_tt2;
    const int per = (G + 31) / 32;
    int loc[8];
    int sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      loc[i] = 0;
      const int gi = lane * per + i;
      if (i < per && gi < G) {
        const int n = s_off[gi + 1] - s_off[gi];
        loc[i] = n > 0 ? ((n + BN - 1) / BN) * nwb : 0;
      }
      sum += loc[i];
    }
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    int run = incl - sum;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int gi = lane * per + i;
      if (i < per && gi < G) s_tt[gi] = run;
      run += loc[i];
    }
    if (lane == 31) s_tt[G] = incl;
  }
  __syncthreads();
  const int total1 = s_tt1[G], total2 = s_tt2[G];
  const int total = total1 + total2;
  if (static_cast<int>(blockIdx.x) >= total) return;

  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<uint32_t*>(s_tmem)), C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  // work item t -> (down?, tile)
  auto item = [&](int t, bool& dn) -> WsTile {
    dn = t >= total1;
    return dn ? ws_tile<BN>(t - total1, total2, s_tt2, s_off, G, nwb2) : ws_tile<BN>(t, total1, s_tt1, s_off, G, nwb1);
  };

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0)
    if (lane == 0) {
      tma_prefetch_desc(&tma_w1);
      tma_prefetch_desc(&tma_x1);
      tma_prefetch_desc(&tma_w2);
      tma_prefetch_desc(&tma_x2);
    }
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    uint32_t armed = 0, armed_ph = 0;
    // readiness of a down item, acquire-loaded one item ahead so that its
    // latency hides behind the current item's loads (stale values only send
    // an item down the wait path)
    auto flag_of = [&](int t) -> int {
      if (t < total1 || t >= total) return 0;
      bool d_;
      const WsTile U = item(t, d_);
      return ld_acquire_gpu(g.ready + U.g);
    };
    int flag_cur = lane == 0 ? flag_of(static_cast<int>(blockIdx.x)) : 0;
    const uint64_t pol_once = policy_evict_first();
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      bool dn;
      const WsTile T = item(t, dn);
      const int flag = flag_cur;
      if (lane == 0) flag_cur = flag_of(t + static_cast<int>(gridDim.x));
      if (lane == 0) {
        const CUtensorMap* tw = dn ? &tma_w2 : &tma_w1;
        const CUtensorMap* tx = dn ? &tma_x2 : &tma_x1;
        const int wrow0 = T.g * (dn ? g.wrows2 : g.wrows1) + T.wb * WS_BM;
        // an expert of one token chunk reads each weight block once: evict-first
        const bool once = s_off[T.g + 1] - s_off[T.g] <= BN;
        const int KB = (dn ? g.kdim2 : g.kdim1) / WS_BK;
        const int nload = (T.ntok + WS_BOX - 1) / WS_BOX;
        const uint32_t bytes = C::A_BYTES + nload * C::BOX_BYTES;
        int pre = 0;  // k-blocks whose weights go out before the dependency is met
        const int need = ((s_off[T.g + 1] - s_off[T.g] + BN - 1) / BN) * nwb1;
        // already met: the ordinary pipeline, weights and h rows together
        const bool met = dn && flag >= need;
        if (met) fence_proxy_async_all();  // h, written by generic stores, read through the tensor map
        if (dn && !met) {
          pre = KB < STAGES ? KB : STAGES;
          const int st0 = stage;
          for (int kb = 0; kb < pre; ++kb) {
            if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(FULL_BAR(stage), bytes);
            if (once)
              tma_load_2d_hint(sA + stage * C::A_BYTES, tw, FULL_BAR(stage), kb * WS_BK, wrow0, pol_once);
            else
              tma_load_2d(sA + stage * C::A_BYTES, tw, FULL_BAR(stage), kb * WS_BK, wrow0);
            armed |= 1u << stage;
            armed_ph = (armed_ph & ~(1u << stage)) | (ph << stage);
            if (++stage == STAGES) {
              stage = 0;
              ph ^= 1u;
            }
          }
          if (ok) {
            // every gate/up item of expert T.g has stored its h slice
            const volatile int32_t* rp = g.ready + T.g;
            const uint64_t t0 = globaltimer_ns();
            while (*rp < need) {
              if (*s_abort || globaltimer_ns() - t0 > g.limit_ns) {
                ok = false;
                break;
              }
            }
            __threadfence();
            fence_proxy_async_all();  // the h rows, written by generic stores, read through the tensor map
          }
          if (ok) {
            int st = st0;
            for (int kb = 0; kb < pre; ++kb) {
              const uint32_t dB = sB + st * C::B_BYTES;
              for (int i = 0; i < nload; ++i)
                tma_load_2d(dB + i * C::BOX_BYTES, tx, FULL_BAR(st), kb * WS_BK, T.row0 + i * WS_BOX);
              if (++st == STAGES) st = 0;
            }
          }
        }
        for (int kb = pre; ok && kb < KB; ++kb) {
          if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(FULL_BAR(stage), bytes);
          if (once)
            tma_load_2d_hint(sA + stage * C::A_BYTES, tw, FULL_BAR(stage), kb * WS_BK, wrow0, pol_once);
          else
            tma_load_2d(sA + stage * C::A_BYTES, tw, FULL_BAR(stage), kb * WS_BK, wrow0);
          const uint32_t dB = sB + stage * C::B_BYTES;
          for (int i = 0; i < nload; ++i)
            tma_load_2d(dB + i * C::BOX_BYTES, tx, FULL_BAR(stage), kb * WS_BK, T.row0 + i * WS_BOX);
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
    }
    if (lane == 0 && !ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      // let the copies this thread started land before the CTA can exit (a
      // stage whose activation rows were never requested runs to the limit)
      int no_abort = 0;
      for (int s = 0; s < STAGES; ++s)
        if ((armed >> s) & 1u) mbar_wait(FULL_BAR(s), (armed_ph >> s) & 1u, g.limit_ns, &no_abort);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------ MMA issuer
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true, issued = false;
    int it = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
      bool dn;
      const WsTile T = item(t, dn);
      const int KB = (dn ? g.kdim2 : g.kdim1) / WS_BK;
      const uint32_t idesc = idesc_bf16_f32(WS_BM, (T.ntok + 15) & ~15);
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait(TEMPTY_BAR(acc), aph ^ 1u, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t dt = tmem_base + static_cast<uint32_t>(acc * BN);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(FULL_BAR(stage), ph, g.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = smem_desc_kmajor<WS_BK>(sA + stage * C::A_BYTES);
        const uint64_t bd = smem_desc_kmajor<WS_BK>(sB + stage * C::B_BYTES);
#pragma unroll
        for (int kk = 0; kk < WS_BK / 16; ++kk)
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
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      if (issued) {
        int no_abort = 0;
        tc_commit(DRAIN_BAR);
        mbar_wait(DRAIN_BAR, 0, g.limit_ns, &no_abort);
      }
    }
  } else if (warp >= 2) {
    // ------------------------------------------------ epilogue (4 warps)
    const int q = warp & 3;  // TMEM lanes [32q, 32q + 32)
    int it = 0;
    int xpar = 0;
    bool ok = true;
    const int et = threadIdx.x - 64;  // 0..127 among the epilogue warps
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
      bool dn;
      const WsTile T = item(t, dn);
      const int acc = it & 1;
      const uint32_t aph = (it >> 1) & 1;
      if (!mbar_wait(TFULL_BAR(acc), aph, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t tb = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      // as k_moe_ws: 32-token chunks through a bf16 tile in shared memory;
      // gate/up items write silu(gate) * up to h (64 features per item),
      // down items write y (128 features per item)
      const int OC = dn ? WS_BM : WS_BM / 2;
      __nv_bfloat16* out = static_cast<__nv_bfloat16*>(dn ? g.y : g.h);
      const int64_t ld = dn ? g.y_ld : g.h_ld;
      const int fbase = T.wb * OC;
#pragma unroll 1
      for (int c0 = 0; c0 < T.ntok; c0 += 32) {
        uint32_t r[32];
        tmem_ld32(tb + c0, r);
        tc_wait_ld();
        __nv_bfloat16* st = stile + xpar * (32 * WS_BM);
        if (!dn) {
          const bool is_gate = q < 2;
          const int pr = q & 1;
          float* xb = xch + (xpar * 2 + pr) * 1024;  // [32 columns][32 lanes]
          if (!is_gate) {
#pragma unroll
            for (int c = 0; c < 32; ++c) xb[c * 32 + lane] = __uint_as_float(r[c]);
          }
          named_bar_sync(1, 128);
          if (is_gate) {
#pragma unroll
            for (int c = 0; c < 32; ++c)
              st[c * OC + pr * 32 + lane] = __float2bfloat16_rn(silu_f(__uint_as_float(r[c])) * xb[c * 32 + lane]);
          }
        } else {
#pragma unroll
          for (int c = 0; c < 32; ++c) st[c * OC + q * 32 + lane] = __float2bfloat16_rn(__uint_as_float(r[c]));
        }
        named_bar_sync(1, 128);
        const int nc = min(32, T.ntok - c0);
        const int VPR = OC / 8;  // 16-byte vectors per token row
        for (int v = et; v < 32 * VPR; v += 128) {
          const int row = v / VPR, cv = v - row * VPR;
          if (row < nc) {
            const uint4 val = *reinterpret_cast<const uint4*>(st + row * OC + cv * 8);
            *reinterpret_cast<uint4*>(out + static_cast<int64_t>(T.row0 + c0 + row) * ld + fbase + cv * 8) = val;
          }
        }
        xpar ^= 1;
      }
      tc_fence_before();
      mbar_arrive(TEMPTY_BAR(acc));
      if (!dn) {
        // this item's h slice is stored: publish it to the down items of T.g
        fence_proxy_async_all();
        named_bar_sync(1, 128);
        if (et == 0) {
          __threadfence();
          atomicAdd(g.ready + T.g, 1);
        }
      }
    }
    if (!ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
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
}

template <int STAGES, int BN>
static int launch_ffn_ws_bn(const void* x_perm, int rows, int d, int m, const void* w_gu, const void* w_down,
                            const int32_t* offsets, int G, void* h, void* y, int32_t* ready, int32_t* status,
                            cudaStream_t s) {
  using C = WsFfnCfg<STAGES, BN>;
  CUtensorMap tw1, tx1, tw2, tx2;
  DM_RET(make_tmap_bf16(&tw1, w_gu, static_cast<uint64_t>(d), static_cast<uint64_t>(G) * 2 * m, WS_BM, WS_BK));
  DM_RET(make_tmap_bf16(&tx1, x_perm, static_cast<uint64_t>(d), static_cast<uint64_t>(rows), WS_BOX, WS_BK));
  DM_RET(make_tmap_bf16(&tw2, w_down, static_cast<uint64_t>(m), static_cast<uint64_t>(G) * d, WS_BM, WS_BK));
  DM_RET(make_tmap_bf16(&tx2, h, static_cast<uint64_t>(m), static_cast<uint64_t>(rows), WS_BOX, WS_BK));
  WsFfnArgs g;
  g.offsets = offsets;
  g.G = G;
  g.rows = rows;
  g.wrows1 = 2 * m;
  g.kdim1 = d;
  g.wrows2 = d;
  g.kdim2 = m;
  g.h = h;
  g.h_ld = m;
  g.y = y;
  g.y_ld = d;
  g.ready = ready;
  g.status = status;
  g.limit_ns = static_cast<uint64_t>(wait_limit_ns());
  auto kern = k_ffn_ws<STAGES, BN>;
  static_assert(C::SMEM <= 232448, "shared memory budget");
  static_assert(C::SMEM > 232448 / 2, "one CTA per SM: the dependency waits need every CTA resident");
  DM_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(C::SMEM)));
  const int64_t ub = (static_cast<int64_t>(rows) / BN + G) * ((2 * m + d) / WS_BM);
  const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(sm_count(), ub)));
  DM_CUDA_CHECK(launch_pdl(kern, dim3(grid), dim3(192), C::SMEM, s, tw1, tx1, tw2, tx2, g));
  return DECOMOE_OK;
}

// Token chunk by row count, as launch_ws_auto.
static int launch_ffn_ws(const void* x_perm, int rows, int d, int m, const void* w_gu, const void* w_down,
                         const int32_t* offsets, int G, void* h, void* y, int32_t* ready, int32_t* status,
                         cudaStream_t s) {
  if (rows <= 256)
    return launch_ffn_ws_bn<ffn_ws_max_stages<32>(), 32>(x_perm, rows, d, m, w_gu, w_down, offsets, G, h, y, ready,
                                                         status, s);
  if (rows <= 512)
    return launch_ffn_ws_bn<ffn_ws_max_stages<64>(), 64>(x_perm, rows, d, m, w_gu, w_down, offsets, G, h, y, ready,
                                                         status, s);
  if (rows <= 1024)
    return launch_ffn_ws_bn<ffn_ws_max_stages<128>(), 128>(x_perm, rows, d, m, w_gu, w_down, offsets, G, h, y,
                                                           ready, status, s);
  return launch_ffn_ws_bn<ffn_ws_max_stages<256>(), 256>(x_perm, rows, d, m, w_gu, w_down, offsets, G, h, y, ready,
                                                         status, s);
}

// ------------------------------------------------------------------ fused prefill FFN
// Gate/up and down of the tokens-as-M path in one persistent launch, with
// k_gemm_tc's tiles (128 rows x 256, 4-stage ring, two TMEM accumulators,
// 8 epilogue warps). Work items: every gate/up tile (tile_coords order),
// then every down tile (same order); static round robin. A down tile of
// M-tile j reads the h rows that the 2m/256 gate/up tiles of j store: those
// bump ready[j] after their stores (release); the down tile issues its
// weight k-blocks first, polls ready[j] (acquire, bounded), then requests the
// h rows. The early CTAs of the down phase start while the last gate/up
// tiles still run, instead of after a launch boundary. Deadlock-free as
// k_ffn_ws (gate/up items never wait; one CTA per SM, grid <= SMs). ready[]
// (one int per M-tile) is zero at launch.
//
// With x set, the launch also performs the dispatch's row gather: each CTA's
// epilogue warps copy, for every gate/up item of the CTA in work order, one
// 1/NT1 share of that item's M-tile rows x_perm[r] = x[perm[r]] and publish
// it (stores, proxy fence, barrier, release add on gathered[M-tile]); they
// copy shares while the accumulator they need next is still being computed. A gate/up item's A rows are requested once all NT1
// shares of its M-tile are in (acquire, bounded; its weight k-blocks go out
// first), as a down item waits for h. The gathers wait on nothing, so this
// adds no cycle; the first wave's rows are in after one share per CTA
// instead of after a separate gather launch.
// Non-blocking: has the phase with this parity completed?
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

struct TcFfnArgs {
  const int32_t* offsets;  // [G + 1]
  int G;
  int rows;
  int d, m;
  void* h;  // [rows, m] bf16
  void* y;  // [rows, d] bf16
  int32_t* ready;
  int32_t* status;
  uint64_t limit_ns;
  const uint4* x;      // gather source [tokens, d / 8] (16-byte vectors), or null: x_perm is filled
  const int32_t* perm;  // [rows] token of each dispatched row
  uint4* x_perm;        // [rows, d / 8], written by the gather
  int32_t* gathered;    // per M-tile: shares copied (zero at launch)
};

constexpr int FFN_BN = 256, FFN_BK = 64, FFN_STAGES = 4, FFN_EW = 8;
using FfnCfg = TcCfg<FFN_BN, FFN_STAGES, FFN_BK, 1, 1>;

__global__ void __launch_bounds__(64 + 32 * FFN_EW, 1)
    k_ffn_tc(const __grid_constant__ CUtensorMap tma_a1, const __grid_constant__ CUtensorMap tma_b1,
             const __grid_constant__ CUtensorMap tma_a2, const __grid_constant__ CUtensorMap tma_b2,
             const TcFfnArgs g) {
  using C = FfnCfg;
  constexpr int BN = FFN_BN, STAGES = FFN_STAGES, EW = FFN_EW;
  __shared__ int s_gperm[C::BM + 1];  // token rows of the share being gathered; [BM]: a broadcast flag
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sA = raw + pad;
  const uint32_t sB = sA + STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
  int* s_off = reinterpret_cast<int*>(bars + C::NBARS);
  int* s_mt = s_off + (C::MAXG + 1);
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(s_mt + (C::MAXG + 1));
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t bar0 = smem_u32(bars);
#define FULL_BAR(s) (bar0 + 8u * (s))
#define EMPTY_BAR(s) (bar0 + 8u * (STAGES + (s)))
#define TFULL_BAR(a) (bar0 + 8u * (2 * STAGES + (a)))
#define TEMPTY_BAR(a) (bar0 + 8u * (2 * STAGES + 2 + (a)))
#define DRAIN_BAR (bar0 + 8u * (2 * STAGES + 4))

  const int G = g.G;
  if (threadIdx.x == 0) {
    *s_abort = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(FULL_BAR(s), 1);
      mbar_init(EMPTY_BAR(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(TFULL_BAR(a), 1);
      mbar_init(TEMPTY_BAR(a), 32 * EW);
    }
    mbar_init(DRAIN_BAR, 1);
    fence_mbar_init();
  }
  pdl_wait();
  for (int i = threadIdx.x; i <= G; i += blockDim.x) s_off[i] = g.offsets[i];
  __syncthreads();
  if (warp == 2) {
    // exclusive scan of M-tiles per group: s_mt[e] = first M-tile of e
    const int per = (G + 31) / 32;  // <= 8
    int loc[8];
    int sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      loc[i] = 0;
      const int gi = lane * per + i;
      if (i < per && gi < G) {
        const int n = s_off[gi + 1] - s_off[gi];
        loc[i] = n > 0 ? (n + C::BM - 1) / C::BM : 0;
      }
      sum += loc[i];
    }
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    int run = incl - sum;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int gi = lane * per + i;
      if (i < per && gi < G) s_mt[gi] = run;
      run += loc[i];
    }
    if (lane == 31) s_mt[G] = incl;
  }
  __syncthreads();
  const int NT1 = 2 * g.m / BN, NT2 = g.d / BN;
  const int total1 = s_mt[G] * NT1, total2 = s_mt[G] * NT2;
  const int total = total1 + total2;
  if (static_cast<int>(blockIdx.x) >= total) return;  // before any TMEM or TMA use

  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<uint32_t*>(s_tmem)), C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  // work item t -> (down?, group, M-tile of the group, N-tile, M-tile index)
  struct Item {
    bool dn;
    int grp, mt, nb, mtg;
  };
  auto item = [&](int t) -> Item {
    Item r;
    r.dn = t >= total1;
    const int tl = r.dn ? t - total1 : t;
    tile_coords(tl, r.dn ? NT2 : NT1, s_mt, G, r.grp, r.mt, r.nb);
    r.mtg = s_mt[r.grp] + r.mt;
    return r;
  };

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0)
    if (lane == 0) {
      tma_prefetch_desc(&tma_a1);
      tma_prefetch_desc(&tma_b1);
      tma_prefetch_desc(&tma_a2);
      tma_prefetch_desc(&tma_b2);
    }
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    uint32_t armed = 0, armed_ph = 0;
    // what an item's A rows wait for: a down item for its M-tile's h, a
    // gate/up item (with the gather) for its M-tile's rows; NT1 counts each.
    // Acquire-loaded one item ahead (as k_ffn_ws).
    auto dep_of = [&](const Item& it) -> const int32_t* {
      return it.dn ? g.ready : (g.x != nullptr ? g.gathered : nullptr);
    };
    auto flag_of = [&](int t) -> int {
      if (t >= total) return 0;
      const Item it = item(t);
      const int32_t* dp = dep_of(it);
      return dp != nullptr ? ld_acquire_gpu(dp + it.mtg) : 0;
    };
    int flag_cur = lane == 0 ? flag_of(static_cast<int>(blockIdx.x)) : 0;
    const uint64_t pol_once = policy_evict_first();
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      const Item it = item(t);
      const int flag = flag_cur;
      if (lane == 0) flag_cur = flag_of(t + static_cast<int>(gridDim.x));
      if (lane == 0) {
        const CUtensorMap* ta = it.dn ? &tma_a2 : &tma_a1;
        const CUtensorMap* tb = it.dn ? &tma_b2 : &tma_b1;
        const int row0 = s_off[it.grp] + it.mt * C::BM;
        const int brow = it.grp * (it.dn ? g.d : 2 * g.m) + it.nb * BN;
        const int KB = (it.dn ? g.m : g.d) / FFN_BK;
        const int32_t* dp = dep_of(it);
        // an expert of one M-tile reads its weights once: they go to L2 as
        // evict-first, leaving room for the weights that later M-tiles reuse
        const bool once = s_mt[it.grp + 1] - s_mt[it.grp] == 1;
        int pre = 0;  // k-blocks whose weights go out before the dependency is met
        // already met (the usual case once the first wave is under way): the
        // ordinary pipeline, A rows and weights together
        const bool met = dp == nullptr || flag >= NT1;
        if (dp != nullptr && met) fence_proxy_async_all();  // rows written by generic stores, read through TMA
        if (!met) {
          pre = KB < STAGES ? KB : STAGES;
          const int st0 = stage;
          for (int kb = 0; kb < pre; ++kb) {
            if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(FULL_BAR(stage), C::A_BYTES + C::B_BYTES);
            if (once)
              tma_load_2d_hint(sB + stage * C::B_BYTES, tb, FULL_BAR(stage), kb * FFN_BK, brow, pol_once);
            else
              tma_load_2d(sB + stage * C::B_BYTES, tb, FULL_BAR(stage), kb * FFN_BK, brow);
            armed |= 1u << stage;
            armed_ph = (armed_ph & ~(1u << stage)) | (ph << stage);
            if (++stage == STAGES) {
              stage = 0;
              ph ^= 1u;
            }
          }
          if (ok) {
            // every gate/up tile of this M-tile has stored its h columns (down
            // item), or every share of its rows is gathered (gate/up item)
            const volatile int32_t* rp = dp + it.mtg;
            const uint64_t t0 = globaltimer_ns();
            while (*rp < NT1) {
              if (*s_abort || globaltimer_ns() - t0 > g.limit_ns) {
                ok = false;
                break;
              }
            }
            __threadfence();
            fence_proxy_async_all();  // rows written by generic stores, read through the tensor map
          }
          if (ok) {
            int st = st0;
            for (int kb = 0; kb < pre; ++kb) {
              tma_load_2d(sA + st * C::A_BYTES, ta, FULL_BAR(st), kb * FFN_BK, row0);
              if (++st == STAGES) st = 0;
            }
          }
        }
        for (int kb = pre; ok && kb < KB; ++kb) {
          if (!mbar_wait(EMPTY_BAR(stage), ph ^ 1u, g.limit_ns, s_abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(FULL_BAR(stage), C::A_BYTES + C::B_BYTES);
          tma_load_2d(sA + stage * C::A_BYTES, ta, FULL_BAR(stage), kb * FFN_BK, row0);
          if (once)
            tma_load_2d_hint(sB + stage * C::B_BYTES, tb, FULL_BAR(stage), kb * FFN_BK, brow, pol_once);
          else
            tma_load_2d(sB + stage * C::B_BYTES, tb, FULL_BAR(stage), kb * FFN_BK, brow);
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
    }
    if (lane == 0 && !ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      int no_abort = 0;
      for (int s = 0; s < STAGES; ++s)
        if ((armed >> s) & 1u) mbar_wait(FULL_BAR(s), (armed_ph >> s) & 1u, g.limit_ns, &no_abort);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------ MMA issuer
    constexpr uint32_t IDESC = idesc_bf16_f32(C::BM, BN);
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true, issued = false;
    int n = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++n) {
      const bool dn = t >= total1;
      const int KB = (dn ? g.m : g.d) / FFN_BK;
      const int acc = n & 1;
      const uint32_t aph = (n >> 1) & 1;
      if (!mbar_wait(TEMPTY_BAR(acc), aph ^ 1u, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t dt = tmem_base + static_cast<uint32_t>(acc * BN);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(FULL_BAR(stage), ph, g.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = smem_desc_kmajor<FFN_BK>(sA + stage * C::A_BYTES);
        const uint64_t bd = smem_desc_kmajor<FFN_BK>(sB + stage * C::B_BYTES);
#pragma unroll
        for (int kk = 0; kk < FFN_BK / 16; ++kk)
          tc_mma_f16(dt, ad + 2u * kk, bd + 2u * kk, IDESC, (kb | kk) != 0 ? 1u : 0u);
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
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
      if (issued) {
        int no_abort = 0;
        tc_commit(DRAIN_BAR);
        mbar_wait(DRAIN_BAR, 0, g.limit_ns, &no_abort);
      }
    }
  } else if (warp >= 2) {
    // ------------------------------------------------ row gather (with g.x):
    // one share of each of this CTA's gate/up M-tiles, in work order, copied
    // while the accumulator the epilogue needs next is still being computed
    const int et = static_cast<int>(threadIdx.x) - 64;  // 0 .. 32*EW-1
    int gshare = g.x != nullptr ? static_cast<int>(blockIdx.x) : total1;  // next share's work item
    auto gather_share = [&](int t) {
      const int vec = g.d / 8;
      constexpr int U = 8;  // 16-byte loads in flight per thread
      const Item it = item(t);
      const int r0 = s_off[it.grp] + it.mt * C::BM;
      const int r1 = min(r0 + C::BM, s_off[it.grp + 1]);
      const int per = (r1 - r0 + NT1 - 1) / NT1;
      const int a = min(r0 + it.nb * per, r1), b = min(a + per, r1);
      for (int i = et; i < b - a; i += 32 * EW) s_gperm[i] = g.perm[a + i];
      named_bar_sync(1, 32 * EW);
      const int nv = (b - a) * vec;
      for (int i0 = et; i0 < nv; i0 += 32 * EW * U) {
        uint4 v[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int i = i0 + u * 32 * EW;
          if (i < nv) {
            const int r = i / vec;
            v[u] = __ldg(g.x + static_cast<int64_t>(s_gperm[r]) * vec + (i - r * vec));
          }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int i = i0 + u * 32 * EW;
          if (i < nv) {
            const int r = i / vec;
            g.x_perm[static_cast<int64_t>(a + r) * vec + (i - r * vec)] = v[u];
          }
        }
      }
      // publish the share to the gate/up tiles of this M-tile (and free
      // s_gperm for the next share)
      fence_proxy_async_all();
      named_bar_sync(1, 32 * EW);
      if (warp == 2 && lane == 0) {
        __threadfence();
        atomicAdd(g.gathered + it.mtg, 1);
      }
    };
    // ------------------------------------------------ epilogue (k_gemm_tc's)
    const int q = warp & 3;
    const int wp = (warp - 2) >> 2;
    constexpr int WPQ = EW / 4;
    bool ok = true;
    int n = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++n) {
      const Item it = item(t);
      const int acc = n & 1;
      const uint32_t aph = (n >> 1) & 1;
      const int row0 = s_off[it.grp] + it.mt * C::BM;
      const int row_end = s_off[it.grp + 1];
      // gather shares until this tile's accumulator is complete (one thread
      // tests the barrier, all epilogue threads follow its answer); while
      // shares remain the warps never block here, so every share gets copied
      while (gshare < total1) {
        if (et == 0) s_gperm[C::BM] = mbar_test(TFULL_BAR(acc), aph) ? 1 : 0;
        named_bar_sync(1, 32 * EW);
        const bool full = s_gperm[C::BM] != 0;
        named_bar_sync(1, 32 * EW);
        if (full) break;
        gather_share(gshare);
        gshare += gridDim.x;
      }
      if (!mbar_wait(TFULL_BAR(acc), aph, g.limit_ns, s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int grow = row0 + q * 32 + lane;
      const bool valid = grow < row_end;
      const uint32_t tb = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      if (!it.dn) {
        constexpr int GU = DECOMOE_GU_BLOCK;
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(g.h);
#pragma unroll 1
        for (int cc = 32 * wp; cc < BN / 2; cc += 32 * WPQ) {
          const int half = cc / GU, c = cc % GU;
          uint32_t gr[32], ur[32];
          tmem_ld32(tb + half * 2 * GU + c, gr);
          tmem_ld32(tb + half * 2 * GU + GU + c, ur);
          tc_wait_ld();
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float g0 = __uint_as_float(gr[2 * i]), g1 = __uint_as_float(gr[2 * i + 1]);
            const float u0 = __uint_as_float(ur[2 * i]), u1 = __uint_as_float(ur[2 * i + 1]);
            pk[i] = pack_bf16x2(silu_f(g0) * u0, silu_f(g1) * u1);
          }
          if (valid) {
            uint4* dst = reinterpret_cast<uint4*>(out + static_cast<int64_t>(grow) * g.m + it.nb * (BN / 2) + cc);
#pragma unroll
            for (int v = 0; v < 4; ++v) dst[v] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
          }
        }
      } else {
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(g.y);
#pragma unroll 1
        for (int c = 32 * wp; c < BN; c += 32 * WPQ) {
          uint32_t r[32];
          tmem_ld32(tb + c, r);
          tc_wait_ld();
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) pk[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
          if (valid) {
            uint4* dst = reinterpret_cast<uint4*>(out + static_cast<int64_t>(grow) * g.d + it.nb * BN + c);
#pragma unroll
            for (int v = 0; v < 4; ++v) dst[v] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
          }
        }
      }
      tc_fence_before();
      mbar_arrive(TEMPTY_BAR(acc));
      if (!it.dn) {
        // this tile's h columns are stored: publish them to the down tiles
        fence_proxy_async_all();
        named_bar_sync(1, 32 * EW);
        if (warp == 2 && lane == 0) {
          __threadfence();
          atomicAdd(g.ready + it.mtg, 1);
        }
      }
    }
    if (!ok) {
      *s_abort = 1;
      report_status(g.status, DECOMOE_ERR_TIMEOUT);
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
}

// gather_x / perm given: the launch fills x_perm itself (see k_ffn_tc);
// the gathered counters follow the ready counters in the same array.
static int launch_ffn_tc(const void* x_perm, int rows, int d, int m, const void* w_gu, const void* w_down,
                         const int32_t* offsets, int G, void* h, void* y, int32_t* ready, int32_t* status,
                         cudaStream_t s, const void* gather_x = nullptr, const int32_t* perm = nullptr) {
  using C = FfnCfg;
  CUtensorMap ta1, tb1, ta2, tb2;
  DM_RET(make_tmap_bf16(&ta1, x_perm, static_cast<uint64_t>(d), static_cast<uint64_t>(rows), C::BM, FFN_BK));
  DM_RET(make_tmap_bf16(&tb1, w_gu, static_cast<uint64_t>(d), static_cast<uint64_t>(G) * 2 * m, FFN_BN, FFN_BK));
  DM_RET(make_tmap_bf16(&ta2, h, static_cast<uint64_t>(m), static_cast<uint64_t>(rows), C::BM, FFN_BK));
  DM_RET(make_tmap_bf16(&tb2, w_down, static_cast<uint64_t>(m), static_cast<uint64_t>(G) * d, FFN_BN, FFN_BK));
  TcFfnArgs g;
  g.offsets = offsets;
  g.G = G;
  g.rows = rows;
  g.d = d;
  g.m = m;
  g.h = h;
  g.y = y;
  g.ready = ready;
  g.status = status;
  g.limit_ns = static_cast<uint64_t>(wait_limit_ns());
  g.x = static_cast<const uint4*>(gather_x);
  g.perm = perm;
  g.x_perm = static_cast<uint4*>(const_cast<void*>(x_perm));
  g.gathered = ready + (rows / C::BM + G + 1);
  static_assert(C::SMEM + sizeof(int) * (C::BM + 1) <= 232448, "shared memory budget");
  static_assert(C::SMEM > 232448 / 2, "one CTA per SM: the dependency waits need every CTA resident");
  DM_CUDA_CHECK(cudaFuncSetAttribute(k_ffn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(C::SMEM)));
  const int64_t ub = (static_cast<int64_t>(rows) / C::BM + G) * static_cast<int64_t>((2 * m + d) / FFN_BN);
  const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(sm_count(), ub)));
  DM_CUDA_CHECK(launch_pdl(k_ffn_tc, dim3(grid), dim3(64 + 32 * FFN_EW), C::SMEM, s, ta1, tb1, ta2, tb2, g));
  return DECOMOE_OK;
}

// X: [rows, kdim] token rows grouped by expert, or with GATHER_B the source
// tensor [x_tensor_rows, kdim] whose row b_rows[r] is token row r;
// W: [G * wrows, kdim].
template <bool SWIGLU, int STAGES, bool GATHER_B = false, int BN = 256>
static int launch_ws(const void* X, int rows, int kdim, const void* W, int wrows, const int32_t* offsets, int G,
                     void* out, int64_t out_ld, int32_t* status, cudaStream_t s, const int32_t* b_rows = nullptr,
                     int64_t x_tensor_rows = 0) {
  using C = WsCfg<STAGES, SWIGLU, BN>;
  constexpr int WS_BN = BN;
  CUtensorMap tw, tx;
  DM_RET(make_tmap_bf16(&tw, W, static_cast<uint64_t>(kdim), static_cast<uint64_t>(G) * wrows, WS_BM, WS_BK));
  if (GATHER_B)
    DM_RET(make_tmap_bf16(&tx, X, static_cast<uint64_t>(kdim), static_cast<uint64_t>(x_tensor_rows), 1, WS_BK));
  else
    DM_RET(make_tmap_bf16(&tx, X, static_cast<uint64_t>(kdim), static_cast<uint64_t>(rows), WS_BOX, WS_BK));
  WsArgs g;
  g.offsets = offsets;
  g.G = G;
  g.rows = rows;
  g.wrows = wrows;
  g.kdim = kdim;
  g.out = out;
  g.out_ld = out_ld;
  g.status = status;
  g.limit_ns = static_cast<uint64_t>(wait_limit_ns());
  g.b_rows = b_rows;
  auto kern = k_moe_ws<SWIGLU, STAGES, GATHER_B, BN>;
  static_assert(C::SMEM <= 232448, "shared memory budget");
  DM_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(C::SMEM)));
  const int64_t ub_tiles = (static_cast<int64_t>(rows) / WS_BN + G) * (wrows / WS_BM);
  const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(sm_count(), ub_tiles)));
  DM_CUDA_CHECK(launch_pdl(kern, dim3(grid), dim3(192), C::SMEM, s, tw, tx, g));
  return DECOMOE_OK;
}

// Weights-stationary launch with the token chunk sized to the row count: an
// expert never gets more rows than there are tokens, and rows = T * k with
// k >= 1, so for rows <= 256 a 32-token chunk usually covers every expert in
// one chunk (decode); smaller chunks buy a deeper weight-streaming ring.
template <bool SWIGLU>
static int launch_ws_auto(const void* X, int rows, int kdim, const void* W, int wrows, const int32_t* offsets,
                          int G, void* out, int64_t out_ld, int32_t* status, cudaStream_t s) {
  if (rows <= 256)
    return launch_ws<SWIGLU, ws_max_stages<SWIGLU, 32>(), false, 32>(X, rows, kdim, W, wrows, offsets, G, out,
                                                                     out_ld, status, s);
  if (rows <= 512)
    return launch_ws<SWIGLU, ws_max_stages<SWIGLU, 64>(), false, 64>(X, rows, kdim, W, wrows, offsets, G, out,
                                                                     out_ld, status, s);
  if (rows <= 1024)
    return launch_ws<SWIGLU, ws_max_stages<SWIGLU, 128>(), false, 128>(X, rows, kdim, W, wrows, offsets, G, out,
                                                                       out_ld, status, s);
  return launch_ws<SWIGLU, 4, false, 256>(X, rows, kdim, W, wrows, offsets, G, out, out_ld, status, s);
}

bool router_tc_supported(int d, int E) { return d % 64 == 0 && (E == 128 || E == 256); }

// Router on the tensor cores with the router rows as the M operand (E = 128
// or 256 rows, one or two M tiles) and the tokens as N tiles of BN columns, so
// that T = 2048 already spreads over 128 CTAs; the epilogue writes the
// transpose, logits[t, e], 32 experts of one token per warp store.
template <int BN>
static int launch_router_bn(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E,
                            float* logits, int32_t* status, cudaStream_t s) {
  const int64_t npad = (T + BN - 1) / BN * BN;
  return launch_tc<BN, EPI_F32_BIAS_T, 8, 64>(w_r, E, d, x, T, nullptr, 1, static_cast<int>(npad), logits, E,
                                              bias, status, s, static_cast<int>(T));
}

int launch_router_tc(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E,
                     float* logits, int32_t* status, cudaStream_t s) {
  if (T > 0x7fffff00LL) {
    set_error("router_logits: T too large for the tensor-core path");
    return DECOMOE_ERR_UNSUPPORTED;
  }
  const int64_t ctas = sm_count();
  if (T <= 16 * ctas) return launch_router_bn<16>(x, w_r, bias, T, d, E, logits, status, s);
  if (T <= 32 * ctas) return launch_router_bn<32>(x, w_r, bias, T, d, E, logits, status, s);
  return launch_router_bn<64>(x, w_r, bias, T, d, E, logits, status, s);
}

// k-split router: KS k slices of the router GEMM write partial logits
// [KS][T][E] (no bias) to the scratch, then k_router_reduce adds the slices in
// slice order and the bias last: logits = (((p0 + p1) + ...) + p_{KS-1}) + b.
// More CTAs with fewer k-blocks each (and N = 64 tokens per MMA instead of
// 16) than the unsplit kernel at the same token count.
template <int KS>
__global__ void __launch_bounds__(256)
    k_router_reduce(const float4* __restrict__ part, int64_t n4, const float* __restrict__ bias, int E,
                    float4* __restrict__ logits) {
  pdl_enter();
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float4 v[KS];
#pragma unroll
    for (int sl = 0; sl < KS; ++sl) v[sl] = __ldcs(part + sl * n4 + i);  // every slice load in flight
    float4 acc = v[0];
#pragma unroll
    for (int sl = 1; sl < KS; ++sl) {
      acc.x += v[sl].x;
      acc.y += v[sl].y;
      acc.z += v[sl].z;
      acc.w += v[sl].w;
    }
    if (bias != nullptr) {
      const int e = static_cast<int>((i * 4) % E);
      acc.x += bias[e];
      acc.y += bias[e + 1];
      acc.z += bias[e + 2];
      acc.w += bias[e + 3];
    }
    logits[i] = acc;
  }
}

int router_split_ks(int64_t T, int d, int E) {
  if (!router_tc_supported(d, E) || d % (64 * 16) != 0) return 1;
  const int64_t tiles = (T + 63) / 64, ctas = sm_count();
  if (tiles * 16 <= ctas) return 16;
  if (tiles * 4 <= ctas) return 4;
  return 1;
}

template <int KS>
static int launch_router_split_ks(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E,
                                  float* logits, float* scratch, int32_t* status, cudaStream_t s) {
  const int64_t npad = (T + 63) / 64 * 64;
  const int64_t n = T * E;
  DM_RET((launch_tc<64, EPI_F32_BIAS_T, 8, 64, 0, 1, 8, 1, KS>(w_r, E, d, x, T, nullptr, 1, static_cast<int>(npad),
                                                               scratch, E, nullptr, status, s, static_cast<int>(T),
                                                               nullptr, 0, nullptr, n)));
  const int64_t n4 = n / 4;
  const int blocks = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>((n4 + 255) / 256, sm_count())));
  DM_CUDA_CHECK(launch_pdl(k_router_reduce<KS>, dim3(blocks), dim3(256), 0, s,
                           reinterpret_cast<const float4*>(scratch), n4, bias, E, reinterpret_cast<float4*>(logits)));
  return DECOMOE_OK;
}

int launch_router_parts(const void* x, const void* w_r, int64_t T, int d, int E, float* scratch, int32_t* status,
                        cudaStream_t s, int* ks_out) {
  const int ks = router_split_ks(T, d, E);
  *ks_out = ks;
  const int64_t npad = (T + 63) / 64 * 64;
  const int64_t n = T * E;
  switch (ks) {
    case 16:
      return launch_tc<64, EPI_F32_BIAS_T, 8, 64, 0, 1, 8, 1, 16>(w_r, E, d, x, T, nullptr, 1, static_cast<int>(npad),
                                                                  scratch, E, nullptr, status, s, static_cast<int>(T),
                                                                  nullptr, 0, nullptr, n);
    case 4:
      return launch_tc<64, EPI_F32_BIAS_T, 8, 64, 0, 1, 8, 1, 4>(w_r, E, d, x, T, nullptr, 1, static_cast<int>(npad),
                                                                 scratch, E, nullptr, status, s, static_cast<int>(T),
                                                                 nullptr, 0, nullptr, n);
    default:
      return DECOMOE_OK;  // no split at this size: nothing launched
  }
}

int launch_router_split(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E, float* logits,
                        float* scratch, int32_t* status, cudaStream_t s) {
  switch (router_split_ks(T, d, E)) {
    case 16: return launch_router_split_ks<16>(x, w_r, bias, T, d, E, logits, scratch, status, s);
    case 4: return launch_router_split_ks<4>(x, w_r, bias, T, d, E, logits, scratch, status, s);
    default: return launch_router_tc(x, w_r, bias, T, d, E, logits, status, s);
  }
}

// ------------------------------------------------------------------ CUDA-core paths
template <typename T>
__device__ __forceinline__ float ld_f(const T* p);
template <>
__device__ __forceinline__ float ld_f<float>(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ld_f<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}
template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ int find_group(const int32_t* __restrict__ offsets, int G, int r) {
  int lo = 0, hi = G - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (offsets[mid] <= r)
      lo = mid;
    else
      hi = mid - 1;
  }
  return lo;
}

// h[r, f] = silu(W_gate[e] x_r)_f * (W_up[e] x_r)_f with the interleaved gate/up
// layout. One thread per (row, feature).
template <typename T>
__global__ void k_simt_gate_up(const T* __restrict__ A, const int32_t* __restrict__ offsets, int G,
                               const T* __restrict__ Wgu, int d, int m, T* __restrict__ H,
                               const int32_t* __restrict__ a_rows) {
  const int rows = offsets[G];
  const int f = blockIdx.x * blockDim.x + threadIdx.x;
  if (f >= m) return;
  for (int r = blockIdx.y; r < rows; r += gridDim.y) {
    const int e = find_group(offsets, G, r);
    const int blk = f / DECOMOE_GU_BLOCK, i = f % DECOMOE_GU_BLOCK;
    const int64_t grow = static_cast<int64_t>(e) * 2 * m + blk * 2 * DECOMOE_GU_BLOCK + i;
    const T* wg = Wgu + grow * d;
    const T* wu = wg + static_cast<int64_t>(DECOMOE_GU_BLOCK) * d;
    const T* x = A + static_cast<int64_t>(a_rows ? a_rows[r] : r) * d;
    float ag = 0.f, au = 0.f;
    for (int j = 0; j < d; ++j) {
      const float xv = ld_f(x + j);
      ag = fmaf(xv, ld_f(wg + j), ag);
      au = fmaf(xv, ld_f(wu + j), au);
    }
    const float hv = ag / (1.0f + expf(-ag)) * au;
    H[static_cast<int64_t>(r) * m + f] = from_f<T>(hv);
  }
}

// y[r, n] = sum_f W_down[e][n, f] h[r, f]. One thread per (row, output).
template <typename T>
__global__ void k_simt_down(const T* __restrict__ H, const int32_t* __restrict__ offsets, int G,
                            const T* __restrict__ Wd, int d, int m, T* __restrict__ Y) {
  const int rows = offsets[G];
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= d) return;
  for (int r = blockIdx.y; r < rows; r += gridDim.y) {
    const int e = find_group(offsets, G, r);
    const T* w = Wd + (static_cast<int64_t>(e) * d + n) * m;
    const T* h = H + static_cast<int64_t>(r) * m;
    float acc = 0.f;
    for (int f = 0; f < m; ++f) acc = fmaf(ld_f(h + f), ld_f(w + f), acc);
    Y[static_cast<int64_t>(r) * d + n] = from_f<T>(acc);
  }
}

// ------------------------------------------------------------------ weight layout
__global__ void k_weight_layout(const uint4* __restrict__ wg, const uint4* __restrict__ wu,
                                uint4* __restrict__ wgu, int E, int m, int vec) {
  const int64_t rows_out = static_cast<int64_t>(E) * 2 * m;
  const int lane = threadIdx.x & 31;
  const int64_t gw = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t ro = gw; ro < rows_out; ro += nw) {
    const int64_t e = ro / (2 * m);
    const int rr = static_cast<int>(ro - e * 2 * m);
    const int blk = rr / (2 * DECOMOE_GU_BLOCK), w = rr % (2 * DECOMOE_GU_BLOCK);
    const bool is_up = w >= DECOMOE_GU_BLOCK;
    const int f = blk * DECOMOE_GU_BLOCK + (is_up ? w - DECOMOE_GU_BLOCK : w);
    const uint4* src = (is_up ? wu : wg) + (e * m + f) * vec;
    uint4* dst = wgu + ro * vec;
    for (int c = lane; c < vec; c += 32) dst[c] = src[c];
  }
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

int decomoe_weight_layout(const void* w_gate, const void* w_up, void* w_gate_up, int E, int d, int m,
                          int dtype, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(w_gate && w_up && w_gate_up, "weight_layout: null pointer");
  DM_ARG_CHECK(E > 0 && d > 0 && m > 0, "weight_layout: bad sizes");
  DM_ARG_CHECK(m % DECOMOE_GU_BLOCK == 0, "weight_layout: m=%d must be a multiple of %d", m, DECOMOE_GU_BLOCK);
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "weight_layout: bad dtype");
  const size_t row_bytes = static_cast<size_t>(d) * dtype_bytes(dtype);
  DM_ARG_CHECK(row_bytes % 16 == 0 && aligned16(w_gate) && aligned16(w_up) && aligned16(w_gate_up),
               "weight_layout: rows must be 16-byte multiples, pointers 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int blocks = sm_count() * 8;
  k_weight_layout<<<blocks, 256, 0, s>>>(static_cast<const uint4*>(w_gate), static_cast<const uint4*>(w_up),
                                         static_cast<uint4*>(w_gate_up), E, m,
                                         static_cast<int>(row_bytes / 16));
  DM_LAUNCH_CHECK("k_weight_layout");
  return DECOMOE_OK;
}

static int expert_check(const char* name, const void* a, const int32_t* offsets, int64_t rows, int K, int d,
                        int m, int dtype, const void* w, void* out) {
  DM_ARG_CHECK(rows >= 0 && rows < 0x7fffffffLL, "%s: rows out of range", name);
  DM_ARG_CHECK(K >= 1 && K <= DECOMOE_MAX_E, "%s: K=%d outside [1, %d]", name, K, DECOMOE_MAX_E);
  DM_ARG_CHECK(d > 0 && m > 0, "%s: bad d/m", name);
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "%s: bad dtype", name);
  DM_ARG_CHECK(m % DECOMOE_GU_BLOCK == 0, "%s: m must be a multiple of %d", name, DECOMOE_GU_BLOCK);
  if (rows == 0) return DECOMOE_OK;
  DM_ARG_CHECK(a && offsets && w && out, "%s: null pointer", name);
  if (dtype == DECOMOE_BF16) {
    // tensor-core tiles: 256 output columns (gate/up interleaved 2m, down d)
    DM_ARG_CHECK(m % 128 == 0, "%s: bf16 needs m %% 128 == 0 (m=%d)", name, m);
    DM_ARG_CHECK(d % 256 == 0, "%s: bf16 needs d %% 256 == 0 (d=%d)", name, d);
    DM_ARG_CHECK(aligned16(a) && aligned16(w) && aligned16(out), "%s: pointers must be 16-byte aligned", name);
  }
  return DECOMOE_OK;
}

// Pipeline shape of the two expert GEMMs: k-block depth (64 -> 128-byte
// swizzle, 32 -> 64-byte swizzle) and the number of shared-memory stages.
#ifndef DECOMOE_GU_BK
#define DECOMOE_GU_BK 64
#endif
#ifndef DECOMOE_GU_STAGES
#define DECOMOE_GU_STAGES 4
#endif
#ifndef DECOMOE_DN_BK
#define DECOMOE_DN_BK 64
#endif
#ifndef DECOMOE_GU_MP
#define DECOMOE_GU_MP 1
#endif
#ifndef DECOMOE_GU_OCC
#define DECOMOE_GU_OCC 1
#endif
#ifndef DECOMOE_DN_OCC
#define DECOMOE_DN_OCC 1
#endif
#ifndef DECOMOE_GU_EW
#define DECOMOE_GU_EW 8
#endif
#ifndef DECOMOE_DN_EW
#define DECOMOE_DN_EW 8
#endif
#ifndef DECOMOE_DN_MP
#define DECOMOE_DN_MP 1
#endif
#ifndef DECOMOE_DN_STAGES
#define DECOMOE_DN_STAGES 4
#endif
constexpr int GU_BK = DECOMOE_GU_BK, GU_STAGES = DECOMOE_GU_STAGES;
constexpr int DN_BK = DECOMOE_DN_BK, DN_STAGES = DECOMOE_DN_STAGES;
constexpr int GU_MP = DECOMOE_GU_MP, DN_MP = DECOMOE_DN_MP;
constexpr int GU_OCC = DECOMOE_GU_OCC, DN_OCC = DECOMOE_DN_OCC, GU_EW = DECOMOE_GU_EW, DN_EW = DECOMOE_DN_EW;

int decomoe_expert_gate_up(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d, int m,
                           int dtype, const void* w_gate_up, void* h, int32_t* status_dev, int32_t* sched_dev,
                           decomoe_stream_t stream) {
  clear_error();
  DM_RET(expert_check("expert_gate_up", x_perm, offsets, rows, K, d, m, dtype, w_gate_up, h));
  if (rows == 0) return DECOMOE_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int R = static_cast<int>(rows);
  if (dtype == DECOMOE_F32) {
    dim3 g1((m + 127) / 128, static_cast<unsigned>(std::min(R, 65535)));
    k_simt_gate_up<float><<<g1, 128, 0, s>>>(static_cast<const float*>(x_perm), offsets, K,
                                              static_cast<const float*>(w_gate_up), d, m, static_cast<float*>(h),
                                              nullptr);
    DM_LAUNCH_CHECK("k_simt_gate_up");
    return DECOMOE_OK;
  }
  if (static_cast<int64_t>(R) <= static_cast<int64_t>(DECOMOE_WS_MAX_AVG_ROWS) * K)
    return launch_ws_auto<true>(x_perm, R, d, w_gate_up, 2 * m, offsets, K, h, m, status_dev, s);
  // A = x_perm [R, d], B = w_gate_up [K*2m, d] (only experts < K are read)
  return launch_tc<256, EPI_SWIGLU, GU_STAGES, GU_BK, false, GU_MP, GU_EW, GU_OCC>(
      x_perm, R, d, w_gate_up, static_cast<int64_t>(K) * 2 * m, offsets, K, 2 * m, h, m, nullptr, status_dev, s, 0,
      nullptr, 0, sched_dev);
}

int decomoe_expert_down(const void* h, const int32_t* offsets, int64_t rows, int K, int d, int m, int dtype,
                        const void* w_down, void* y_perm, int32_t* status_dev, int32_t* sched_dev,
                        decomoe_stream_t stream) {
  clear_error();
  DM_RET(expert_check("expert_down", h, offsets, rows, K, d, m, dtype, w_down, y_perm));
  if (rows == 0) return DECOMOE_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int R = static_cast<int>(rows);
  if (dtype == DECOMOE_F32) {
    dim3 g2((d + 127) / 128, static_cast<unsigned>(std::min(R, 65535)));
    k_simt_down<float><<<g2, 128, 0, s>>>(static_cast<const float*>(h), offsets, K,
                                           static_cast<const float*>(w_down), d, m, static_cast<float*>(y_perm));
    DM_LAUNCH_CHECK("k_simt_down");
    return DECOMOE_OK;
  }
  if (static_cast<int64_t>(R) <= static_cast<int64_t>(DECOMOE_WS_MAX_AVG_ROWS) * K)
    return launch_ws_auto<false>(h, R, m, w_down, d, offsets, K, y_perm, d, status_dev, s);
  // A = h [R, m], B = w_down [K*d, m]
  return launch_tc<256, EPI_BF16, DN_STAGES, DN_BK, false, DN_MP, DN_EW, DN_OCC>(h, R, m, w_down, static_cast<int64_t>(K) * d, offsets,
                                                                  K, d, y_perm, d, nullptr, status_dev, s, 0,
                                                                  nullptr, 0, sched_dev);
}

int decomoe_expert_gate_up_gather(const void* x, int64_t T, const int32_t* perm_token, const int32_t* offsets,
                                  int64_t rows, int K, int d, int m, int dtype, const void* w_gate_up, void* h,
                                  int32_t* status_dev, int32_t* sched_dev, decomoe_stream_t stream) {
  (void)sched_dev;  // the gathered form keeps the static tile order
  clear_error();
  DM_RET(expert_check("expert_gate_up_gather", x, offsets, rows, K, d, m, dtype, w_gate_up, h));
  if (rows == 0) return DECOMOE_OK;
  DM_ARG_CHECK(perm_token != nullptr && T > 0 && T < 0x7fffffffLL, "expert_gate_up_gather: bad perm_token or T");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int R = static_cast<int>(rows);
  if (dtype == DECOMOE_F32) {
    dim3 g1((m + 127) / 128, static_cast<unsigned>(std::min(R, 65535)));
    k_simt_gate_up<float><<<g1, 128, 0, s>>>(static_cast<const float*>(x), offsets, K,
                                              static_cast<const float*>(w_gate_up), d, m, static_cast<float*>(h),
                                              perm_token);
    DM_LAUNCH_CHECK("k_simt_gate_up");
    return DECOMOE_OK;
  }
  if (static_cast<int64_t>(R) <= static_cast<int64_t>(DECOMOE_WS_MAX_AVG_ROWS) * K)
    return launch_ws<true, 4, true>(x, R, d, w_gate_up, 2 * m, offsets, K, h, m, status_dev, s, perm_token, T);
  return launch_tc<256, EPI_SWIGLU, GU_STAGES, GU_BK, 2>(
      x, R, d, w_gate_up, static_cast<int64_t>(K) * 2 * m, offsets, K, 2 * m, h, m, nullptr, status_dev, s, 0,
      perm_token, T);
}

int decomoe_expert_swiglu_gather(const void* x, int64_t T, const int32_t* perm_token, const int32_t* offsets,
                                 int64_t rows, int K, int d, int m, int dtype, const void* w_gate_up,
                                 const void* w_down, void* h_ws, void* y_perm, int32_t* status_dev,
                                 int32_t* sched_dev, decomoe_stream_t stream) {
  DM_RET(decomoe_expert_gate_up_gather(x, T, perm_token, offsets, rows, K, d, m, dtype, w_gate_up, h_ws,
                                       status_dev, sched_dev, stream));
  return decomoe_expert_down(h_ws, offsets, rows, K, d, m, dtype, w_down, y_perm, status_dev, sched_dev, stream);
}

int decomoe_expert_swiglu(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d, int m,
                          int dtype, const void* w_gate_up, const void* w_down, void* h_ws, void* y_perm,
                          int32_t* status_dev, int32_t* sched_dev, decomoe_stream_t stream) {
  DM_RET(decomoe_expert_gate_up(x_perm, offsets, rows, K, d, m, dtype, w_gate_up, h_ws, status_dev, sched_dev,
                                stream));
  return decomoe_expert_down(h_ws, offsets, rows, K, d, m, dtype, w_down, y_perm, status_dev, sched_dev, stream);
}

// Reference CUDA-core path for bf16 (same math as the tensor-core path: bf16
// products, fp32 accumulation, h rounded to bf16). Not part of the public
// header; used by tests to localise disagreements between the tensor-core
// kernels and the oracle.
int decomoe_expert_swiglu_ref(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d, int m,
                               const void* w_gate_up, const void* w_down, void* h_ws, void* y_perm,
                               decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(rows >= 0 && rows < 0x7fffffffLL && K >= 1 && K <= DECOMOE_MAX_E && d > 0 && m > 0,
               "expert_swiglu_ref: bad sizes");
  if (rows == 0) return DECOMOE_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int R = static_cast<int>(rows);
  dim3 g1((m + 127) / 128, static_cast<unsigned>(std::min(R, 65535)));
  k_simt_gate_up<__nv_bfloat16><<<g1, 128, 0, s>>>(static_cast<const __nv_bfloat16*>(x_perm), offsets, K,
                                                    static_cast<const __nv_bfloat16*>(w_gate_up), d, m,
                                                    static_cast<__nv_bfloat16*>(h_ws), nullptr);
  DM_LAUNCH_CHECK("k_simt_gate_up<bf16>");
  dim3 g2((d + 127) / 128, static_cast<unsigned>(std::min(R, 65535)));
  k_simt_down<__nv_bfloat16><<<g2, 128, 0, s>>>(static_cast<const __nv_bfloat16*>(h_ws), offsets, K,
                                                 static_cast<const __nv_bfloat16*>(w_down), d, m,
                                                 static_cast<__nv_bfloat16*>(y_perm));
  DM_LAUNCH_CHECK("k_simt_down<bf16>");
  return DECOMOE_OK;
}

}  // extern "C"

namespace decomoe {

// Rows from which the fused launch is taken (with fewer, the gate/up tiles
// leave SMs idle and the fused form gains nothing), and up to which the
// tokens-as-M form is fused (measured per layer: 7 us faster at 2048 and
// 16384 rows, 1-2 us at 8192 and 32768, 5 and 20 us slower at 65536 and
// 131072 rows).
#ifndef DECOMOE_FFN_FUSED_MIN_ROWS
#define DECOMOE_FFN_FUSED_MIN_ROWS 16
#endif
#ifndef DECOMOE_FFN_FUSED_TC_MAX_ROWS
#define DECOMOE_FFN_FUSED_TC_MAX_ROWS 32768
#endif
// Both expert GEMMs in one launch: k_ffn_ws at decode sizes (bf16, at most 8
// rows per expert on average), k_ffn_tc above up to
// DECOMOE_FFN_FUSED_TC_MAX_ROWS rows; nothing launched (and *launched false)
// for fp32, fewer than DECOMOE_FFN_FUSED_MIN_ROWS rows or more than that.
// Which one-launch form the expert FFN takes: FFN_FUSED_NONE (two launches),
// FFN_FUSED_WS (decode sizes) or FFN_FUSED_TC (tokens as M).
int expert_ffn_fused_kind(int64_t rows, int K, int m, int dtype) {
  constexpr int64_t min_rows = DECOMOE_FFN_FUSED_MIN_ROWS;
  constexpr int64_t tc_max_rows = DECOMOE_FFN_FUSED_TC_MAX_ROWS;
  if (dtype != DECOMOE_BF16 || rows < min_rows || rows <= 0 || K <= 0) return FFN_FUSED_NONE;
  if (rows <= static_cast<int64_t>(DECOMOE_WS_MAX_AVG_ROWS) * K) return FFN_FUSED_WS;
  // the tokens-as-M kernel tiles gate/up in whole 256-column blocks
  if (rows > tc_max_rows || (2 * m) % FFN_BN != 0) return FFN_FUSED_NONE;
  return FFN_FUSED_TC;
}

int launch_expert_ffn_fused(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d, int m, int dtype,
                            const void* w_gate_up, const void* w_down, void* h, void* y_perm, int32_t* ready,
                            int32_t* status, cudaStream_t s, bool* launched, const void* gather_x,
                            const int32_t* perm) {
  *launched = false;
  const int kind = expert_ffn_fused_kind(rows, K, m, dtype);
  DM_ARG_CHECK(gather_x == nullptr || kind == FFN_FUSED_TC, "expert ffn: the row gather needs the tokens-as-M form");
  if (kind == FFN_FUSED_NONE) return DECOMOE_OK;
  DM_RET(expert_check("expert_gate_up", x_perm, offsets, rows, K, d, m, dtype, w_gate_up, h));
  DM_RET(expert_check("expert_down", h, offsets, rows, K, d, m, dtype, w_down, y_perm));
  DM_ARG_CHECK(ready != nullptr, "expert ffn: null ready counters");
  if (gather_x != nullptr)
    DM_ARG_CHECK(perm != nullptr && aligned16(gather_x), "expert ffn: gather needs perm and a 16-byte aligned x");
  if (kind == FFN_FUSED_WS)
    DM_RET(launch_ffn_ws(x_perm, static_cast<int>(rows), d, m, w_gate_up, w_down, offsets, K, h, y_perm, ready,
                         status, s));
  else
    DM_RET(launch_ffn_tc(x_perm, static_cast<int>(rows), d, m, w_gate_up, w_down, offsets, K, h, y_perm, ready,
                         status, s, gather_x, perm));
  *launched = true;
  return DECOMOE_OK;
}

// int32 counters the fused expert launch needs (zero at launch): one per
// expert (decode kernel) or two per M-tile (prefill kernel: h stored, rows
// gathered).
size_t expert_ffn_sync_ints(int64_t rows, int E) { return 2 * static_cast<size_t>(rows / 128 + E + 1); }

}  // namespace decomoe

extern "C" {

size_t decomoe_expert_swiglu_ready_ints(int64_t rows, int K) {
  return rows < 0 || K <= 0 ? 0 : decomoe::expert_ffn_sync_ints(rows, K);
}

int decomoe_expert_swiglu_fused(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d, int m,
                                int dtype, const void* w_gate_up, const void* w_down, void* h_ws, void* y_perm,
                                int32_t* ready, int32_t* status_dev, decomoe_stream_t stream) {
  using namespace decomoe;
  clear_error();
  bool fused = false;
  DM_RET(launch_expert_ffn_fused(x_perm, offsets, rows, K, d, m, dtype, w_gate_up, w_down, h_ws, y_perm, ready,
                                 status_dev, reinterpret_cast<cudaStream_t>(stream), &fused));
  if (fused) return DECOMOE_OK;
  return decomoe_expert_swiglu(x_perm, offsets, rows, K, d, m, dtype, w_gate_up, w_down, h_ws, y_perm, status_dev,
                               nullptr, stream);
}

int decomoe_expert_swiglu_fused_gather(const void* x, int64_t T, const int32_t* perm_token, const int32_t* offsets,
                                       int64_t rows, int K, int d, int m, int dtype, const void* w_gate_up,
                                       const void* w_down, void* x_perm, void* h_ws, void* y_perm, int32_t* ready,
                                       int32_t* status_dev, decomoe_stream_t stream) {
  using namespace decomoe;
  clear_error();
  DM_ARG_CHECK(x != nullptr && perm_token != nullptr && T >= 0, "expert_swiglu_fused_gather: null pointer");
  DM_ARG_CHECK(expert_ffn_fused_kind(rows, K, m, dtype) == FFN_FUSED_TC,
               "expert_swiglu_fused_gather: %lld rows at K=%d take no one-launch tokens-as-M form",
               (long long)rows, K);
  bool fused = false;
  DM_RET(launch_expert_ffn_fused(x_perm, offsets, rows, K, d, m, dtype, w_gate_up, w_down, h_ws, y_perm, ready,
                                 status_dev, reinterpret_cast<cudaStream_t>(stream), &fused, x, perm_token));
  return fused ? DECOMOE_OK : DECOMOE_ERR_UNSUPPORTED;
}

}  // extern "C"
