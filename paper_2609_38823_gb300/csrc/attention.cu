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
// Decode sizes (few queries per KV head): one launch of split-key blocks on
// warp-level tensor-core products, the splits of a head merged through the
// shared memory of their thread-block cluster (below). Prefill sizes: a
// transpose of V, then the tcgen05 flash-style kernel (further below).
#include <atomic>
#include <cfloat>

#include "decomoe_internal.cuh"

namespace decomoe {

constexpr int ATT_D = 128;
constexpr int ATT_MAXQ = 64;                    // queries per KV head taken by the decode kernel
constexpr int ATT_PROW = ATT_D + 4;             // floats per partial row: acc[D], m, l, 2 unused (16-byte rows)

// ------------------------------------------------------------------ decode sizes
// Few queries per KV head (a decode step over the cache, or a short chunk):
// block (split s, KV head g, query tile group z) streams keys
// [s * kps, (s + 1) * kps) of head g through a three-chunk TMA ring of 128
// keys (128-byte swizzled 64-feature halves; rows past C read as zero) and
// runs the online softmax of up to 32 of the group's
// nq = n * Hq / Hkv queries on the tensor cores with warp-level
// mma.m16n8k16 (bf16 in, fp32 accumulate): per 16 keys a warp computes
// S = Q K^T for 16 query rows, turns the scores into bf16 weights in
// registers (the accumulator layout of one product is the operand layout of
// the next) and adds P V into its output tile. The eight warps of a block take
// 16 keys of each chunk apiece; their states are merged in warp order into
// the block's partial (m, l, unnormalised output) per query. The splits of
// one (KV head, query tile group) form one thread-block cluster: each block
// pushes its partial of query row r into the shared memory of block
// r % nsplit (distributed shared-memory stores, fire and forget), one cluster
// barrier (release / acquire) makes them visible, and block r then merges
// its rows over the blocks in rank order from its own shared memory and
// stores the output. A barrier split around the launch's start (arrive
// first thing, wait before the first push) keeps pushes out of blocks that
// are not running yet; after the second barrier no block touches another's
// shared memory, so blocks leave freely. A long cache (more than four chunks
// per block with one cluster per head) is split over S clusters per head
// where the SMs allow: each cluster stores its merged (m, l, output) rows in
// a workspace and a second small launch, allowed to be scheduled from this
// launch's start, merges the S clusters in cluster order. No counters, and
// the result does not depend on timing.
constexpr int ATD_WARPS = 8;
constexpr int ATD_CH = 16 * ATD_WARPS;          // keys per staged chunk (16 per warp)
constexpr int ATD_THREADS = 32 * ATD_WARPS;
constexpr int ATD_ROW = ATT_D * 2 + 16;         // padded query row (bytes): conflict-free ldmatrix
constexpr int ATD_QT = 2;                       // 16-row query tiles per block (at most)
constexpr int ATD_HALF = ATD_CH * 64 * 2;       // 128 keys x 64 features, 128-byte swizzle (16 KB)
constexpr int ATD_STAGE = 4 * ATD_HALF;         // K and V halves of one chunk
constexpr int ATD_NST = 3;                      // chunks in flight
// Partial rows pushed into a block by the blocks of its cluster: row r of
// the query tile goes to block r % nsplit, slot (r / nsplit) * nsplit +
// sender rank, so ceil(rows / nsplit) * nsplit <= rows + 15 slots
// (nsplit <= 16).
constexpr int ATD_RSLOTS = ATD_QT * 16 + 15;
constexpr int ATD_RECV = ATD_RSLOTS * ATT_PROW * 4;
constexpr size_t ATD_SMEM =
    1024 + static_cast<size_t>(ATD_NST) * ATD_STAGE + ATD_QT * 16 * ATD_ROW + ATD_RECV + 8 * ATD_NST + 16;
static_assert(ATD_SMEM <= 232448, "decode attention shared memory");
constexpr int ATD_OROW = ATT_D + 8;             // floats per row of the warp merge (conflict-free float2 stores)
static_assert(ATD_WARPS * ATD_QT * 16 * (ATD_OROW + 2) * 4 <= ATD_NST * ATD_STAGE, "warp merge fits in the ring");

struct AttDecArgs {
  const uint4* q;   // [n, Hq, D] (K and V [C, Hkv, D] come through the tensor maps)
  int64_t n, C;
  int Hq, Hkv, kps; // keys per block; a cluster (grid.x) is a run of the head's splits
  int S;            // clusters per (KV head, query tile group): grid.y = Hkv * S
  float sl2;        // scale * log2(e)
  __nv_bfloat16* out;
  float* part;      // S > 1: [Hkv][nz][S][QT * 16][ATT_PROW] merged rows of each cluster
  int32_t* status;
  uint64_t limit_ns;
};

__device__ __forceinline__ float att_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// Four 8x8 bf16 matrices from shared memory; thread t gives the address of
// row t % 8 of matrix t / 8 and receives (row t / 4, columns 2 (t % 4), +1)
// of each (with .trans: of each matrix transposed).
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address of the same shared-memory location in block `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_dsmem_v4(uint32_t addr, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
               : "memory");
}
__device__ __forceinline__ void st_dsmem_v2(uint32_t addr, float x, float y) {
  asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(addr), "f"(x), "f"(y) : "memory");
}
// Split cluster barrier, every thread of every block: arrive (relaxed: no
// ordering) and the matching wait; arrive with release and wait with
// acquire: writes before the arrive (shared, distributed shared and global)
// are visible to the cluster's blocks after the wait.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_release() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait_acquire() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// D (16x8 fp32) += A (16x16 bf16, row) * B (16x8 bf16, col)
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <int QT>
__global__ void __launch_bounds__(ATD_THREADS)
    k_attn_dec(const __grid_constant__ CUtensorMap tma_k, const __grid_constant__ CUtensorMap tma_v,
               const AttDecArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* sKV = smem_raw + pad;                                 // [NST]{K lo, K hi, V lo, V hi}
  uint8_t* sQ = sKV + ATD_NST * ATD_STAGE;                       // [QT * 16][ROW]
  float* s_recv = reinterpret_cast<float*>(sQ + ATD_QT * 16 * ATD_ROW);  // [RSLOTS][PROW]
  uint64_t* bars = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(s_recv) + ATD_RECV);
  volatile int* s_abort = reinterpret_cast<volatile int*>(bars + ATD_NST);
  const uint32_t sKVa = smem_u32(sKV);
  const uint32_t bar0 = smem_u32(bars);
  const int s = blockIdx.x, g = static_cast<int>(blockIdx.y) / a.S, cset = static_cast<int>(blockIdx.y) % a.S;
  const int G = a.Hq / a.Hkv;
  const int nq = static_cast<int>(a.n) * G;
  const int qbase = static_cast<int>(blockIdx.z) * ATD_QT * 16;  // first query row of this block
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int grp = lane >> 2, tig = lane & 3;
  constexpr int VPR = ATT_D / 8;  // 16-byte vectors per head row
  const int64_t k0 = static_cast<int64_t>(cset * static_cast<int>(gridDim.x) + s) * a.kps;
  const int64_t k1 = k0 + a.kps < a.C ? k0 + a.kps : a.C;
  const int nch = k1 > k0 ? static_cast<int>((k1 - k0 + ATD_CH - 1) / ATD_CH) : 0;  // a split past C: none
  if (tid == 0) {
    *s_abort = 0;
    for (int st = 0; st < ATD_NST; ++st) mbar_init(bar0 + 8u * st, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tma_k);
    tma_prefetch_desc(&tma_v);
  }
  __syncthreads();
  // first half of the barrier that keeps pushes out of blocks not yet
  // running (its wait comes before the first push)
  cluster_arrive_relaxed();
  // several clusters per head: the merge launch may be scheduled now (its
  // griddepcontrol.wait still waits for this grid's completion)
  if (a.S > 1) pdl_trigger();
  pdl_wait();  // q, K and V are ready
  // chunk c into stage st: K and V, features 0-63 and 64-127 (keys past C read as zero)
  auto issue = [&](int c, int st) {
    const uint32_t bar = bar0 + 8u * st;
    const uint32_t base = sKVa + st * ATD_STAGE;
    const int key0 = static_cast<int>(k0) + c * ATD_CH;
    mbar_arrive_expect_tx(bar, ATD_STAGE);
    tma_load_3d(base, &tma_k, bar, 0, g, key0);
    tma_load_3d(base + ATD_HALF, &tma_k, bar, 64, g, key0);
    tma_load_3d(base + 2 * ATD_HALF, &tma_v, bar, 0, g, key0);
    tma_load_3d(base + 3 * ATD_HALF, &tma_v, bar, 64, g, key0);
  };
  // query rows (zero rows past the group's queries), requested ahead of the
  // key and value chunks so that they do not queue behind them
  for (int i = tid; i < QT * 16 * VPR; i += ATD_THREADS) {
    const int r = i / VPR, c = i - r * VPR;
    const int qi = qbase + r;
    uint8_t* dst = sQ + r * ATD_ROW + c * 16;
    if (qi < nq) {
      const int ti = qi / G, hj = qi - ti * G;
      cp_async16(smem_u32(dst), a.q + (static_cast<int64_t>(ti) * a.Hq + g * G + hj) * VPR + c);
    } else {
      *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
    }
  }
  int issued = nch < ATD_NST ? nch : ATD_NST;  // chunks whose copies were requested (thread 0)
  if (tid == 0)
    for (int c = 0; c < issued; ++c) issue(c, c);
  cp_async_wait_all();
  __syncthreads();  // the query rows are in place

  // last visible key of this thread's two rows in each query tile
  int64_t lim[QT][2];
#pragma unroll
  for (int qt = 0; qt < QT; ++qt)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int qi = qbase + qt * 16 + grp + 8 * h;
      lim[qt][h] = qi < nq ? a.C - a.n + qi / G : a.C - 1;
    }
  float m[QT][2], l[QT][2], o[QT][16][4];
#pragma unroll
  for (int qt = 0; qt < QT; ++qt) {
    m[qt][0] = m[qt][1] = -INFINITY;
    l[qt][0] = l[qt][1] = 0.f;
#pragma unroll
    for (int j = 0; j < 16; ++j) o[qt][j][0] = o[qt][j][1] = o[qt][j][2] = o[qt][j][3] = 0.f;
  }
  const uint32_t sQa = smem_u32(sQ);
  bool ok = true;
  int c_fail = nch;  // first chunk whose wait ran out
  for (int c = 0; c < nch; ++c) {
    const int buf = c % ATD_NST;
    ok = ok && __all_sync(0xffffffffu, mbar_wait(bar0 + 8u * buf, (c / ATD_NST) & 1, a.limit_ns, s_abort));
    if (!ok && c_fail == nch) c_fail = c;
    const uint32_t sKa = sKVa + buf * ATD_STAGE;  // K halves; V halves follow
    const uint32_t sVa = sKa + 2 * ATD_HALF;
    const int64_t kw = k0 + static_cast<int64_t>(c) * ATD_CH + 16 * warp;  // this warp's first key
    if (ok && kw < k1) {
      // S = Q K^T for this warp's 16 keys (two 8-key n-tiles), per query tile
      float sc[QT][2][4];
#pragma unroll
      for (int qt = 0; qt < QT; ++qt)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) sc[qt][nt][0] = sc[qt][nt][1] = sc[qt][nt][2] = sc[qt][nt][3] = 0.f;
      const int mi = lane >> 3, rr = lane & 7;
#pragma unroll
      for (int ks = 0; ks < ATT_D / 16; ++ks) {
        uint32_t b00, b01, b10, b11;  // n-tile 0 (keys 0-7) and 1 (keys 8-15), features ks*16 + 0-7 / 8-15
        {
          const int key = 16 * warp + (mi >> 1) * 8 + rr, f = ks * 16 + (mi & 1) * 8;
          ldsm_x4(sKa + (f >> 6) * ATD_HALF + key * 128 + ((((f & 63) >> 3) ^ (key & 7)) << 4), b00, b01, b10, b11);
        }
#pragma unroll
        for (int qt = 0; qt < QT; ++qt) {
          uint32_t a0, a1, a2, a3;
          ldsm_x4(sQa + (qt * 16 + (mi & 1) * 8 + rr) * ATD_ROW + (ks * 16 + (mi >> 1) * 8) * 2, a0, a1, a2, a3);
          mma_bf16_16816(sc[qt][0], a0, a1, a2, a3, b00, b01);
          mma_bf16_16816(sc[qt][1], a0, a1, a2, a3, b10, b11);
        }
      }
      // online softmax (log2 units), weights packed as the A operand of P V
      uint32_t pa[QT][4];
#pragma unroll
      for (int qt = 0; qt < QT; ++qt) {
        float t[2][4];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int64_t kp = kw + nt * 8 + 2 * tig + (e & 1);
            const bool vis = kp < k1 && kp <= lim[qt][e >> 1];
            t[nt][e] = vis ? sc[qt][nt][e] * a.sl2 : -INFINITY;
          }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          float mx = fmaxf(fmaxf(t[0][2 * h], t[0][2 * h + 1]), fmaxf(t[1][2 * h], t[1][2 * h + 1]));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
          const float mn = fmaxf(m[qt][h], mx);
          float alpha = 1.f;
          if (mn == -INFINITY) {  // nothing visible yet in this row
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) t[nt][2 * h] = t[nt][2 * h + 1] = 0.f;
          } else {
            alpha = att_ex2(m[qt][h] - mn);
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
              t[nt][2 * h] = att_ex2(t[nt][2 * h] - mn);
              t[nt][2 * h + 1] = att_ex2(t[nt][2 * h + 1] - mn);
            }
            m[qt][h] = mn;
          }
          l[qt][h] = fmaf(l[qt][h], alpha, (t[0][2 * h] + t[0][2 * h + 1]) + (t[1][2 * h] + t[1][2 * h + 1]));
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            o[qt][j][2 * h] *= alpha;
            o[qt][j][2 * h + 1] *= alpha;
          }
        }
        pa[qt][0] = pack_bf16x2(t[0][0], t[0][1]);  // row grp,     keys 2 tig, +1
        pa[qt][1] = pack_bf16x2(t[0][2], t[0][3]);  // row grp + 8
        pa[qt][2] = pack_bf16x2(t[1][0], t[1][1]);  // row grp,     keys 8 + 2 tig, +1
        pa[qt][3] = pack_bf16x2(t[1][2], t[1][3]);  // row grp + 8
      }
      // O += P V: V rows are keys, so the B operand comes through ldmatrix.trans
#pragma unroll
      for (int j = 0; j < ATT_D / 16; ++j) {
        uint32_t v00, v01, v10, v11;  // features 16j + 0-7 (keys 0-7, 8-15), 16j + 8-15 (keys 0-7, 8-15)
        {
          const int key = 16 * warp + (mi & 1) * 8 + rr, f = 16 * j + (mi >> 1) * 8;
          ldsm_x4_t(sVa + (f >> 6) * ATD_HALF + key * 128 + ((((f & 63) >> 3) ^ (key & 7)) << 4), v00, v01, v10,
                    v11);
        }
#pragma unroll
        for (int qt = 0; qt < QT; ++qt) {
          mma_bf16_16816(o[qt][2 * j], pa[qt][0], pa[qt][1], pa[qt][2], pa[qt][3], v00, v01);
          mma_bf16_16816(o[qt][2 * j + 1], pa[qt][0], pa[qt][1], pa[qt][2], pa[qt][3], v10, v11);
        }
      }
    }
    __syncthreads();  // every warp is done with this stage
    if (tid == 0 && ok && c + ATD_NST < nch) {
      issue(c + ATD_NST, buf);
      ++issued;
    }
  }
  if (!ok) {
    // a stage never arrived: record it, let the copies still in flight land
    // (bounded), and finish without results; the cluster barriers below still
    // meet
    *s_abort = 1;
    if (tid == 0) {
      report_status(a.status, DECOMOE_ERR_TIMEOUT);
      int no_abort = 0;
      for (int c = c_fail; c < issued; ++c) mbar_wait(bar0 + 8u * (c % ATD_NST), (c / ATD_NST) & 1, a.limit_ns, &no_abort);
    }
  }
  __syncthreads();

  // merge the warps (warp order) through shared memory: per warp and valid
  // row m, l and the 128 output columns
  const int rv = min(ATD_QT * 16, nq - qbase);  // this block's query rows (>= 1)
  float* sm_o = reinterpret_cast<float*>(sKV);                   // [WARPS][QT*16][OROW]
  float* sm_m = sm_o + ATD_WARPS * ATD_QT * 16 * ATD_OROW;        // [WARPS][QT*16]
  float* sm_l = sm_m + ATD_WARPS * ATD_QT * 16;
#pragma unroll
  for (int qt = 0; qt < QT; ++qt)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float ls = l[qt][h];
      ls += __shfl_xor_sync(0xffffffffu, ls, 1);
      ls += __shfl_xor_sync(0xffffffffu, ls, 2);
      const int r = qt * 16 + grp + 8 * h;
      if (r < rv) {
        if (tig == 0) {
          sm_m[warp * ATD_QT * 16 + r] = m[qt][h];
          sm_l[warp * ATD_QT * 16 + r] = ls;
        }
        float* orow = sm_o + (warp * ATD_QT * 16 + r) * ATD_OROW;
#pragma unroll
        for (int j = 0; j < 16; ++j)
          *reinterpret_cast<float2*>(orow + 8 * j + 2 * tig) = make_float2(o[qt][j][2 * h], o[qt][j][2 * h + 1]);
      }
    }
  __syncthreads();
  // this block's partial rows (m in log2 units, l, unnormalised output), one
  // (row, 4 columns) piece per thread summed over the warps in warp order,
  // pushed into the shared memory of the row's owner, block r % nsplit
  cluster_wait_acquire();  // every block of the cluster is running
  const uint32_t nsplit = gridDim.x;
  const uint32_t rank = cluster_ctarank();
  const uint32_t recv_a = smem_u32(s_recv);
  for (int it = tid; it < rv * (ATT_D / 4); it += ATD_THREADS) {
    const int r = it / (ATT_D / 4), c4 = it - r * (ATT_D / 4);
    float mw[ATD_WARPS], lw[ATD_WARPS];
    float4 ow[ATD_WARPS];
#pragma unroll
    for (int w = 0; w < ATD_WARPS; ++w) {  // every load in flight at once
      mw[w] = sm_m[w * ATD_QT * 16 + r];
      lw[w] = sm_l[w * ATD_QT * 16 + r];
      ow[w] = *reinterpret_cast<const float4*>(sm_o + (w * ATD_QT * 16 + r) * ATD_OROW + 4 * c4);
    }
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < ATD_WARPS; ++w) M = fmaxf(M, mw[w]);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    float L = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < ATD_WARPS; ++w) {
        const float ww = mw[w] == -INFINITY ? 0.f : att_ex2(mw[w] - M);
        acc.x = fmaf(ww, ow[w].x, acc.x);
        acc.y = fmaf(ww, ow[w].y, acc.y);
        acc.z = fmaf(ww, ow[w].z, acc.z);
        acc.w = fmaf(ww, ow[w].w, acc.w);
        L = fmaf(ww, lw[w], L);
      }
    }
    const uint32_t owner = static_cast<uint32_t>(r) % nsplit;
    const uint32_t slot = (static_cast<uint32_t>(r) / nsplit) * nsplit + rank;
    const uint32_t dst = mapa_shared(recv_a + slot * (ATT_PROW * 4), owner);
    st_dsmem_v4(dst + 16u * c4, acc);
    if (c4 == 0) st_dsmem_v2(dst + ATT_D * 4, M, L);
  }
  cluster_arrive_release();
  cluster_wait_acquire();  // every block's rows are in their owners' shared memory
  // block `rank` merges its rows rank, rank + nsplit, ... over the blocks in
  // rank order (threads 0-127 and 128-255: two rows per pass, one column each)
  for (int r0 = static_cast<int>(rank); r0 < rv; r0 += 2 * static_cast<int>(nsplit)) {
    const int r = r0 + (tid >> 7) * static_cast<int>(nsplit);
    const int col = tid & (ATT_D - 1);
    if (r < rv) {
      const float* base = s_recv + (r / static_cast<int>(nsplit)) * static_cast<int>(nsplit) * ATT_PROW;
      constexpr int MAXS = 16;  // cluster size limit
      float mt[MAXS], at[MAXS], lt[MAXS];
#pragma unroll
      for (int t = 0; t < MAXS; ++t) {  // every load in flight at once
        const float* row = base + t * ATT_PROW;
        mt[t] = t < static_cast<int>(nsplit) ? row[ATT_D] : -INFINITY;
        at[t] = t < static_cast<int>(nsplit) ? row[col] : 0.f;
        lt[t] = t < static_cast<int>(nsplit) ? row[ATT_D + 1] : 0.f;
      }
      float M = -INFINITY;
#pragma unroll
      for (int t = 0; t < MAXS; ++t) M = fmaxf(M, mt[t]);
      float acc = 0.f, L = 0.f;
#pragma unroll
      for (int t = 0; t < MAXS; ++t) {
        if (t < static_cast<int>(nsplit)) {
          const float w = mt[t] == -INFINITY ? 0.f : att_ex2(mt[t] - M);  // a split with no visible key weighs 0
          acc = fmaf(w, at[t], acc);
          L = fmaf(w, lt[t], L);
        }
      }
      const int qi = qbase + r;
      if (a.S == 1) {
        const int ti = qi / G, hj = qi - ti * G;
        a.out[(static_cast<int64_t>(ti) * a.Hq + g * G + hj) * ATT_D + col] = __float2bfloat16_rn(acc / L);
      } else {
        // this cluster's merged row, for the merge launch
        float* pr = a.part + ((static_cast<int64_t>(g * gridDim.z + blockIdx.z) * a.S + cset) * (QT * 16) + r) * ATT_PROW;
        pr[col] = acc;
        if (col == 0) {
          pr[ATT_D] = M;
          pr[ATT_D + 1] = L;
        }
      }
    }
  }
  if (a.S == 1) pdl_trigger();
}

// The S <= ATT_MAX_SETS clusters of a (KV head g = blockIdx.x, query tile
// group z = blockIdx.y) merged in cluster order; block blockIdx.z takes two
// of the rows (threads 0-127 and 128-255, one output column each), with all
// S partials' loads in flight at once.
constexpr int ATT_MAX_SETS = 16;
__global__ void __launch_bounds__(ATD_THREADS)
    k_attn_dec_merge(const float* __restrict__ part, int S, int rows, int64_t n, int Hq, int Hkv,
                     __nv_bfloat16* __restrict__ out) {
  pdl_wait();
  const int g = blockIdx.x, z = blockIdx.y, tid = threadIdx.x;
  const int G = Hq / Hkv;
  const int nq = static_cast<int>(n) * G;
  const int r = static_cast<int>(blockIdx.z) * 2 + (tid >> 7), col = tid & (ATT_D - 1);
  const int qi = z * rows + r;
  if (r < rows && qi < nq) {
    const float* base = part + (static_cast<int64_t>(g * gridDim.y + z) * S * rows + r) * ATT_PROW;
    float mc[ATT_MAX_SETS], ac[ATT_MAX_SETS], lc[ATT_MAX_SETS];
#pragma unroll
    for (int c = 0; c < ATT_MAX_SETS; ++c) {
      const float* row = base + static_cast<int64_t>(c) * rows * ATT_PROW;
      mc[c] = c < S ? __ldcg(row + ATT_D) : -INFINITY;
      ac[c] = c < S ? __ldcg(row + col) : 0.f;
      lc[c] = c < S ? __ldcg(row + ATT_D + 1) : 0.f;
    }
    float M = -INFINITY;
#pragma unroll
    for (int c = 0; c < ATT_MAX_SETS; ++c) M = fmaxf(M, mc[c]);
    float acc = 0.f, L = 0.f;
#pragma unroll
    for (int c = 0; c < ATT_MAX_SETS; ++c) {
      if (c < S) {
        const float w = mc[c] == -INFINITY ? 0.f : att_ex2(mc[c] - M);  // a cluster with no visible key weighs 0
        acc = fmaf(w, ac[c], acc);
        L = fmaf(w, lc[c], L);
      }
    }
    const int ti = qi / G, hj = qi - ti * G;
    out[(static_cast<int64_t>(ti) * Hq + g * G + hj) * ATT_D + col] = __float2bfloat16_rn(acc / L);
  }
  pdl_trigger();
}

static int att_max_cluster();
static int att_active_clusters(int cs);
static int att_nz(int64_t nq) { return static_cast<int>((nq + ATD_QT * 16 - 1) / (ATD_QT * 16)); }
// The split of a head's keys: S clusters of at most cs blocks each. One
// cluster per (KV head, query tile group), of the largest size (16, 8, 4) of
// which that many clusters are resident at once, while that streams at most
// four chunks per block; a longer cache takes the cluster size and S that
// put the most blocks to work with every cluster resident at once (the
// device's limit on active clusters of that size) and each block keeping at
// least two chunks.
struct AttPlan {
  int cs, S;
};
static AttPlan att_plan(int64_t C, int Hkv, int nz) {
  const int maxc = att_max_cluster();
  const int64_t sets = static_cast<int64_t>(Hkv) * nz;
  int cs1 = maxc;
  for (int cs : {16, 8, 4})
    if (cs <= maxc && sets <= att_active_clusters(cs)) {
      cs1 = cs;
      break;
    }
  if (C <= static_cast<int64_t>(cs1) * ATD_CH * 4) return {cs1, 1};
  AttPlan best = {cs1, 1};
  int64_t best_blocks = cs1;
  for (int cs : {16, 8, 4}) {
    if (cs > maxc) continue;
    const int64_t by_res = att_active_clusters(cs) / sets;
    const int64_t by_keys = C / (static_cast<int64_t>(cs) * ATD_CH * 2);
    const int64_t S = std::min<int64_t>({by_res, by_keys, static_cast<int64_t>(ATT_MAX_SETS)});
    if (S >= 1 && S * cs > best_blocks) {
      best = {cs, static_cast<int>(S)};
      best_blocks = S * cs;
    }
  }
  return best;
}
// Keys per block, in whole chunks, for the plan's cs * S splits.
static int64_t att_kps(int64_t C, const AttPlan& pl) {
  const int64_t nsplit = std::max<int64_t>(1, std::min<int64_t>((C + ATD_CH - 1) / ATD_CH, pl.cs)) * pl.S;
  int64_t kps = (C + nsplit - 1) / nsplit;
  return (kps + ATD_CH - 1) / ATD_CH * ATD_CH;
}

// Largest cluster of decode blocks this device schedules (16 where the
// non-portable size fits, else the portable 8), per device ordinal.
static std::atomic<int> g_att_cluster[64];
static int att_max_cluster() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 8;
  int v = g_att_cluster[dev].load();
  if (v != 0) return v;
  v = 8;
  bool ok = true;
  for (auto kern : {k_attn_dec<1>, k_attn_dec<2>}) {
    ok = ok && cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(ATD_SMEM)) ==
                   cudaSuccess;
    ok = ok && cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
  }
  if (ok) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(16, 1, 1);
    cfg.blockDim = dim3(ATD_THREADS);
    cfg.dynamicSmemBytes = ATD_SMEM;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 16;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n1 = 0, n2 = 0;
    if (cudaOccupancyMaxActiveClusters(&n1, k_attn_dec<1>, &cfg) == cudaSuccess &&
        cudaOccupancyMaxActiveClusters(&n2, k_attn_dec<2>, &cfg) == cudaSuccess && n1 >= 1 && n2 >= 1)
      v = 16;
  }
  cudaGetLastError();  // a refused query leaves no error behind
  g_att_cluster[dev].store(v);
  return v;
}

// Clusters of cs decode blocks the device keeps resident at once (per device
// ordinal and cluster size 4, 8 or 16; 0 when the query is refused).
static std::atomic<int> g_att_active[64][3];
static int att_active_clusters(int cs) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int slot = cs == 4 ? 0 : cs == 8 ? 1 : 2;
  int v = g_att_active[dev][slot].load();
  if (v != 0) return v > 0 ? v : 0;
  att_max_cluster();  // sets the kernels' shared-memory and cluster-size attributes
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(cs), 1, 1);
  cfg.blockDim = dim3(ATD_THREADS);
  cfg.dynamicSmemBytes = ATD_SMEM;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(cs);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n1 = 0, n2 = 0;
  if (cudaOccupancyMaxActiveClusters(&n1, k_attn_dec<1>, &cfg) != cudaSuccess ||
      cudaOccupancyMaxActiveClusters(&n2, k_attn_dec<2>, &cfg) != cudaSuccess)
    n1 = n2 = 0;
  cudaGetLastError();  // a refused query leaves no error behind
  v = std::min(n1, n2);
  g_att_active[dev][slot].store(v > 0 ? v : -1);
  return v > 0 ? v : 0;
}

// ------------------------------------------------------------------ prefill (tensor cores)
// Many queries per KV head (the compacted sequence's prefill): flash-style
// attention on tcgen05. A CTA takes one tile of 128 query rows for two query
// heads of the same KV group, so each K and V block it streams serves both.
// Per block j of 64 keys and head x: S_x = Q_x K_j^T (M = 128 queries, N = 64
// keys, K = 128 features) into tensor memory; four warps per head (one query
// row per thread) take the row maximum, write p = 2^(s*scale*log2e - m) as
// bf16 into tensor memory (the A operand of the next product) and add p to
// the row sum l; then O_x += P_x V_j (N = 128 features, K = 64 keys, V
// transposed beforehand so that the B operand is K-major) accumulates in
// tensor memory. The reference maximum m of a row moves only when the block
// maximum exceeds it by more than 8 (a factor 256): then that row's O and l
// are scaled by 2^(m_old - m_new) before the next product (otherwise p stays
// below 256, well inside bf16 and fp32); the final output is O / l either
// way. Tensor-core work of one head overlaps the other head's softmax: the
// issue order is PV_0(j), S_0(j+1), PV_1(j), S_1(j+1). Warp 0 streams K_j and
// V_j^T blocks by TMA into a four-stage ring; warp 1 issues the MMAs. Every
// wait is bounded; on a timeout the CTA records DECOMOE_ERR_TIMEOUT, lets its
// copies and MMAs land, frees its tensor memory and returns.
constexpr int ATP_BM = 128;                 // query rows per CTA
constexpr int ATP_BN = 64;                  // keys per block
constexpr int ATP_HEADS = 2;                // query heads per CTA (same KV head)
constexpr int ATP_NST = 4;                  // K / V ring stages
constexpr int ATP_QHALF = 128 * 64 * 2;     // Q: 128 rows x 64 features, 128-byte swizzle (16 KB)
constexpr int ATP_KHALF = ATP_BN * 64 * 2;  // K block: 64 keys x 64 features (8 KB)
constexpr int ATP_VT = 128 * ATP_BN * 2;    // V^T block: 128 features x 64 keys (16 KB)
constexpr int ATP_STAGE = 2 * ATP_KHALF + ATP_VT;
constexpr int ATP_THREADS = 64 + ATP_HEADS * 128;
constexpr int ATP_TMEM_COLS = 512;          // per head: S [0,64), P [64,96), O [128,256)
constexpr float ATP_RESCALE = 8.0f;         // log2 of the largest unnormalised p
constexpr size_t ATP_SMEM = 1024 + ATP_HEADS * 2 * ATP_QHALF + ATP_NST * ATP_STAGE + 32 * 8 + 16;

struct AttPreArgs {
  int64_t n, C;        // queries (the last n positions), keys
  int Hq, group;       // query heads, query heads per KV head
  float scale_log2;    // scale * log2(e)
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

// D(tmem) (+)= A(tmem) * B(smem desc)^T: A is 128 rows (lanes) x 16 bf16
// (8 columns, two elements per 32-bit column, the lower index in the low half).
__device__ __forceinline__ void tc_mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// Values loaded by tcgen05.ld are defined only after tcgen05.wait::ld: route
// them through an empty asm placed after the wait so no use moves above it.
template <int N>
__device__ __forceinline__ void after_wait(uint32_t (&r)[N]) {
#pragma unroll
  for (int i = 0; i < N; ++i) asm volatile("" : "+r"(r[i]));
}
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(ATP_THREADS, 1)
    k_attn_prefill(const __grid_constant__ CUtensorMap tma_q, const __grid_constant__ CUtensorMap tma_k,
                   const __grid_constant__ CUtensorMap tma_vt, const AttPreArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sQ = raw + pad;                              // [head][feature half]
  const uint32_t sKV = sQ + ATP_HEADS * 2 * ATP_QHALF;        // [stage]{K half 0, K half 1, V^T}
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + ATP_HEADS * 2 * ATP_QHALF + ATP_NST * ATP_STAGE);
  volatile uint32_t* s_tmem = reinterpret_cast<volatile uint32_t*>(bars + 32);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  const uint32_t bar0 = smem_u32(bars);
  const uint32_t Q_BAR = bar0, DRAIN = bar0 + 8;
  auto S_FULL = [&](int x) { return bar0 + 16u + 8u * x; };
  auto P_FULL = [&](int x) { return bar0 + 32u + 8u * x; };
  auto O_FINAL = [&](int x) { return bar0 + 48u + 8u * x; };
  auto FULL = [&](int st) { return bar0 + 64u + 8u * st; };
  auto EMPTY = [&](int st) { return bar0 + 96u + 8u * st; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int npair = a.Hq / ATP_HEADS;
  const int ntile = static_cast<int>((a.n + ATP_BM - 1) / ATP_BM);
  // heaviest tiles (most key blocks) first
  const int hp = blockIdx.x % npair;
  const int qt = ntile - 1 - static_cast<int>(blockIdx.x / npair);
  const int h0 = hp * ATP_HEADS;
  const int g = h0 / a.group;  // both heads read KV head g (the group size is even)
  const int64_t p0 = a.C - a.n + static_cast<int64_t>(qt) * ATP_BM;  // position of the tile's first row
  const int64_t last = p0 + ATP_BM - 1 < a.C - 1 ? p0 + ATP_BM - 1 : a.C - 1;
  const int nblk = static_cast<int>(last / ATP_BN) + 1;  // key blocks any row of the tile can see

  if (threadIdx.x == 0) {
    *s_abort = 0;
    mbar_init(Q_BAR, 1);
    mbar_init(DRAIN, 1);
    for (int x = 0; x < ATP_HEADS; ++x) {
      mbar_init(S_FULL(x), 1);
      mbar_init(P_FULL(x), 128);
      mbar_init(O_FINAL(x), 1);
    }
    for (int st = 0; st < ATP_NST; ++st) {
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
  auto S_TM = [&](int x) { return tmem + 256u * x; };
  auto P_TM = [&](int x) { return tmem + 256u * x + 64u; };
  auto O_TM = [&](int x) { return tmem + 256u * x + 128u; };
  constexpr uint32_t IDESC_S = idesc_bf16_f32(ATP_BM, ATP_BN);
  constexpr uint32_t IDESC_O = idesc_bf16_f32(ATP_BM, ATT_D);

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (lane 0)
    if (lane == 0) {
      tma_prefetch_desc(&tma_q);
      tma_prefetch_desc(&tma_k);
      tma_prefetch_desc(&tma_vt);
      bool ok = true;
      uint32_t armed = 0, armed_ph = 0;
      mbar_arrive_expect_tx(Q_BAR, ATP_HEADS * 2 * ATP_QHALF);
      const int qrow0 = qt * ATP_BM;
      for (int x = 0; x < ATP_HEADS; ++x)
        for (int kb = 0; kb < 2; ++kb) tma_load_3d(sQ + (2 * x + kb) * ATP_QHALF, &tma_q, Q_BAR, 64 * kb, h0 + x, qrow0);
      for (int j = 0; j < nblk; ++j) {
        const int st = j % ATP_NST;
        const uint32_t ph = (j / ATP_NST) & 1;
        if (!mbar_wait(EMPTY(st), ph ^ 1u, a.limit_ns, s_abort)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(FULL(st), ATP_STAGE);
        const int key0 = j * ATP_BN;
        const uint32_t base = sKV + st * ATP_STAGE;
        tma_load_3d(base, &tma_k, FULL(st), 0, g, key0);
        tma_load_3d(base + ATP_KHALF, &tma_k, FULL(st), 64, g, key0);
        tma_load_3d(base + 2 * ATP_KHALF, &tma_vt, FULL(st), key0, 0, g);
        armed |= 1u << st;
        armed_ph = (armed_ph & ~(1u << st)) | (ph << st);
      }
      if (!ok) {
        *s_abort = 1;
        report_status(a.status, DECOMOE_ERR_TIMEOUT);
        int no_abort = 0;
        mbar_wait(Q_BAR, 0, a.limit_ns, &no_abort);
        for (int st = 0; st < ATP_NST; ++st)
          if ((armed >> st) & 1u) mbar_wait(FULL(st), (armed_ph >> st) & 1u, a.limit_ns, &no_abort);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (lane 0)
    if (lane == 0) {
      // S_x = Q_x K^T over the 128 features (two 64-feature halves)
      auto issue_s = [&](int x, int st) {
        const uint32_t base = sKV + st * ATP_STAGE;
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint64_t ad = smem_desc_kmajor<64>(sQ + (2 * x + kb) * ATP_QHALF);
          const uint64_t bd = smem_desc_kmajor<64>(base + kb * ATP_KHALF);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_f16(S_TM(x), ad + 2u * kk, bd + 2u * kk, IDESC_S, (kb | kk) != 0 ? 1u : 0u);
        }
      };
      // O_x += P_x V_j over the block's 64 keys
      auto issue_pv = [&](int x, int st, bool acc) {
        const uint64_t bd = smem_desc_kmajor<64>(sKV + st * ATP_STAGE + 2 * ATP_KHALF);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_f16_ts(O_TM(x), P_TM(x) + 8u * kk, bd + 2u * kk, IDESC_O, (acc || kk > 0) ? 1u : 0u);
      };
      bool ok = mbar_wait(Q_BAR, 0, a.limit_ns, s_abort) && mbar_wait(FULL(0), 0, a.limit_ns, s_abort);
      bool issued = false;
      if (ok) {
        tc_fence_after();
        for (int x = 0; x < ATP_HEADS; ++x) {
          issue_s(x, 0);
          tc_commit(S_FULL(x));
        }
        issued = true;
      }
      for (int j = 0; ok && j < nblk; ++j) {
        const int st = j % ATP_NST;
        for (int x = 0; x < ATP_HEADS; ++x) {
          if (!mbar_wait(P_FULL(x), j & 1, a.limit_ns, s_abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_pv(x, st, j > 0);
          if (x == ATP_HEADS - 1) tc_commit(EMPTY(st));  // K_j and V_j read by every product
          if (j + 1 < nblk) {
            const int st1 = (j + 1) % ATP_NST;
            if (x == 0) {
              if (!mbar_wait(FULL(st1), ((j + 1) / ATP_NST) & 1, a.limit_ns, s_abort)) {
                ok = false;
                break;
              }
              tc_fence_after();
            }
            issue_s(x, st1);
            tc_commit(S_FULL(x));
          } else {
            tc_commit(O_FINAL(x));
          }
        }
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
    // ------------------------------------------------ softmax rows
    const int x = (warp - 2) >> 2;          // head of this warp
    const int q = warp & 3;                 // tensor-memory lane quarter of this warp
    const int r = q * 32 + lane;            // query row of the tile
    const int64_t climit = a.C - 1;
    const int64_t qlim = p0 + r < climit ? p0 + r : climit;                    // last visible key of the row
    const int64_t wlim = p0 + q * 32 < climit ? p0 + q * 32 : climit;          // smallest of the warp's rows
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const float sl2 = a.scale_log2;
    float m = 0.f, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nblk; ++j) {
      if (!__all_sync(0xffffffffu, mbar_wait(S_FULL(x), j & 1, a.limit_ns, s_abort))) {  // warp-uniform loads
        ok = false;
        break;
      }
      tc_fence_after();
      const int64_t key0 = static_cast<int64_t>(j) * ATP_BN;
      uint32_t sv[ATP_BN];
      tmem_ld32(S_TM(x) + lane_off, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
      tmem_ld32(S_TM(x) + lane_off + 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
      tc_wait_ld();
      after_wait(sv);
      if (key0 + ATP_BN - 1 > wlim) {  // the causal edge or the end of the keys crosses this warp's rows
        const int64_t d = qlim - key0;
        const int lim = d < 0 ? -1 : static_cast<int>(d);  // d < 64 here
#pragma unroll
        for (int c = 0; c < ATP_BN; ++c)
          if (c > lim) sv[c] = __float_as_uint(-INFINITY);
      }
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int c = 0; c < ATP_BN; ++c) mx[c & 3] = fmaxf(mx[c & 3], __uint_as_float(sv[c]));
      const float m_blk = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * sl2;
      float factor = 1.0f;
      if (j == 0) {
        m = m_blk;  // key 0 is visible to every row
      } else if (m_blk > m + ATP_RESCALE) {
        factor = ex2_approx(m - m_blk);
        m = m_blk;
        l *= factor;
      }
      if (__any_sync(0xffffffffu, factor != 1.0f)) {
        // the previous product into O has completed (S_FULL is committed after it)
#pragma unroll
        for (int c = 0; c < ATT_D / 32; ++c) {
          uint32_t ov[32];
          tmem_ld32(O_TM(x) + lane_off + 32 * c, ov);
          tc_wait_ld();
          after_wait(ov);
#pragma unroll
          for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * factor);
          tmem_st32(O_TM(x) + lane_off + 32 * c, ov);
        }
      }
      float ls[4] = {0.f, 0.f, 0.f, 0.f};
      uint32_t pk[32];
#pragma unroll
      for (int c = 0; c < ATP_BN; c += 2) {
        const float e0 = ex2_approx(fmaf(__uint_as_float(sv[c]), sl2, -m));
        const float e1 = ex2_approx(fmaf(__uint_as_float(sv[c + 1]), sl2, -m));
        ls[(c >> 1) & 3] += e0 + e1;
        pk[c >> 1] = pack_bf16x2(e0, e1);
      }
      l += (ls[0] + ls[1]) + (ls[2] + ls[3]);
      tmem_st32(P_TM(x) + lane_off, pk);
      tc_wait_st();
      tc_fence_before();
      mbar_arrive(P_FULL(x));
    }
    if (ok && __all_sync(0xffffffffu, mbar_wait(O_FINAL(x), 0, a.limit_ns, s_abort))) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int64_t row = static_cast<int64_t>(qt) * ATP_BM + r;
      uint4* dst = reinterpret_cast<uint4*>(a.out + (row * a.Hq + h0 + x) * ATT_D);
#pragma unroll
      for (int c = 0; c < ATT_D / 32; ++c) {
        uint32_t ov[32];
        tmem_ld32(O_TM(x) + lane_off + 32 * c, ov);
        tc_wait_ld();
        after_wait(ov);
        if (row < a.n) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float* o = reinterpret_cast<const float*>(&ov[8 * u]);
            dst[4 * c + u] = make_uint4(pack_bf16x2(o[0] * inv, o[1] * inv), pack_bf16x2(o[2] * inv, o[3] * inv),
                                        pack_bf16x2(o[4] * inv, o[5] * inv), pack_bf16x2(o[6] * inv, o[7] * inv));
          }
        }
      }
    } else {
      *s_abort = 1;
      report_status(a.status, DECOMOE_ERR_TIMEOUT);
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
  // decode sizes: a cluster's splits merge through its shared memory; several
  // clusters per head (long caches) leave their merged rows here
  const int nq = static_cast<int>(n) * (Hq / Hkv);
  const int nz = att_nz(nq);
  const int S = att_plan(C, Hkv, nz).S;
  const int rows = (nq <= 16 ? 1 : 2) * 16;
  return S == 1 ? 0 : align_up(static_cast<size_t>(Hkv) * nz * S * rows * ATT_PROW * 4, 256);
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
  if (need > 0 && (ws == nullptr || ws_bytes < need)) {
    set_error("attention: workspace needs %zu bytes", need);
    return DECOMOE_ERR_WORKSPACE;
  }
  DM_ARG_CHECK(need == 0 || aligned16(ws), "attention: workspace must be 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const float sc = scale > 0.f ? scale : 1.0f / sqrtf(static_cast<float>(D));
  if (att_use_prefill(n, Hq, Hkv)) {
    DM_ARG_CHECK(G % ATP_HEADS == 0, "attention: prefill sizes need an even number of query heads per KV head (%d)",
                 G);
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
    const uint32_t bq[3] = {64, 1, ATP_BM}, bk[3] = {64, 1, ATP_BN}, bv[3] = {ATP_BN, ATT_D, 1};
    DM_RET(make_tmap_bf16_3d(&tq, q, dq, sq, bq));
    DM_RET(make_tmap_bf16_3d(&tk, k_cache, dk, sk, bk));
    DM_RET(make_tmap_bf16_3d(&tv, vt, dv, sv, bv));
    AttPreArgs pa;
    pa.n = n;
    pa.C = C;
    pa.Hq = Hq;
    pa.group = G;
    pa.scale_log2 = sc * 1.4426950408889634f;
    pa.out = static_cast<__nv_bfloat16*>(out);
    pa.status = status_dev;
    pa.limit_ns = static_cast<uint64_t>(wait_limit_ns());
    const int64_t ntile = (n + ATP_BM - 1) / ATP_BM;
    DM_ARG_CHECK(ntile * (Hq / ATP_HEADS) < 0x7fffffffLL, "attention: too many query tiles");
    DM_CUDA_CHECK(cudaFuncSetAttribute(k_attn_prefill, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(ATP_SMEM)));
    DM_CUDA_CHECK(launch_pdl(k_attn_prefill, dim3(static_cast<unsigned>(ntile * (Hq / ATP_HEADS))), dim3(ATP_THREADS),
                             ATP_SMEM, s,
                             tq, tk, tv, pa));
    return DECOMOE_OK;
  }
  AttDecArgs a;
  a.q = static_cast<const uint4*>(q);
  a.n = n;
  a.C = C;
  a.Hq = Hq;
  a.Hkv = Hkv;
  const int nq = static_cast<int>(n) * G;
  const int nz = att_nz(nq);
  const AttPlan pl = att_plan(C, Hkv, nz);
  const int S = pl.S;
  const int64_t kps = att_kps(C, pl);
  DM_ARG_CHECK(kps <= 0x7fffffffLL, "attention: C=%lld keys is too long", (long long)C);
  a.kps = static_cast<int>(kps);
  a.S = S;
  a.part = static_cast<float*>(ws);
  // blocks per cluster (<= pl.cs); with S > 1 the last blocks may find no
  // key left (they weigh 0 in the merge)
  const int nsplit = static_cast<int>((C + kps * S - 1) / (kps * S));
  // the receive slots of the pushed partial rows are sized for clusters of
  // at most 16 blocks (att_plan never picks more)
  if (nsplit < 1 || nsplit > 16) {
    set_error("attention: internal split of %d blocks per cluster (at most 16)", nsplit);
    return DECOMOE_ERR_UNSUPPORTED;
  }
  a.sl2 = sc * 1.4426950408889634f;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.status = status_dev;
  a.limit_ns = static_cast<uint64_t>(wait_limit_ns());
  CUtensorMap tk, tv;  // [C][Hkv][D]: boxes of 128 keys x 64 features of one head
  const uint64_t dkv[3] = {static_cast<uint64_t>(D), static_cast<uint64_t>(Hkv), static_cast<uint64_t>(C)};
  const uint64_t skv[2] = {static_cast<uint64_t>(D) * 2, static_cast<uint64_t>(Hkv) * D * 2};
  const uint32_t bkv[3] = {64, 1, ATD_CH};
  DM_RET(make_tmap_bf16_3d(&tk, k_cache, dkv, skv, bkv));
  DM_RET(make_tmap_bf16_3d(&tv, v_cache, dkv, skv, bkv));
  const dim3 grid(static_cast<unsigned>(nsplit), static_cast<unsigned>(Hkv * S), static_cast<unsigned>(nz));
  auto go = [&](auto kern) -> int {
    DM_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(ATD_SMEM)));
    if (nsplit > 8) DM_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(ATD_THREADS);
    cfg.dynamicSmemBytes = ATD_SMEM;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;  // one cluster per (KV head, query tile group)
    attr[0].val.clusterDim.x = static_cast<unsigned>(nsplit);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    // at most one block per SM: scheduled while the previous kernel drains,
    // waiting on griddepcontrol.wait before it reads q, K or V
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed =
        pdl_enabled(static_cast<int64_t>(grid.x) * grid.y * grid.z) ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    DM_CUDA_CHECK(cudaLaunchKernelEx(&cfg, kern, tk, tv, a));
    if (S > 1)
      DM_CUDA_CHECK(launch_pdl(k_attn_dec_merge,
                               dim3(static_cast<unsigned>(Hkv), static_cast<unsigned>(nz), (nq <= 16 ? 1 : 2) * 8),
                               dim3(ATD_THREADS), 0, s, static_cast<const float*>(ws), S, (nq <= 16 ? 1 : 2) * 16, n,
                               Hq, Hkv, static_cast<__nv_bfloat16*>(out)));
    return DECOMOE_OK;
  };
  return nq <= 16 ? go(k_attn_dec<1>) : go(k_attn_dec<2>);
}

}  // extern "C"
