// Internal helpers shared by the CUDA translation units of libdecomoe:
// error plumbing, launch checks, and inline-PTX wrappers for mbarrier, TMA
// (cp.async.bulk.tensor) and the 5th-generation tensor cores (tcgen05 + TMEM)
// of sm_103a.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <climits>
#include <cstdarg>
#include <cstdio>

#include "../../include/decomoe.h"

namespace decomoe {

// ---------------------------------------------------------------- host side

void set_error(const char* fmt, ...);
void clear_error();
int64_t wait_limit_ns();

#define DM_ARG_CHECK(cond, ...)                  \
  do {                                           \
    if (!(cond)) {                               \
      ::decomoe::set_error(__VA_ARGS__);         \
      return DECOMOE_ERR_INVALID_ARG;            \
    }                                            \
  } while (0)

#define DM_CUDA_CHECK(expr)                                                        \
  do {                                                                             \
    cudaError_t e_ = (expr);                                                       \
    if (e_ != cudaSuccess) {                                                       \
      ::decomoe::set_error("%s: %s (%s:%d)", #expr, cudaGetErrorString(e_),        \
                           __FILE__, __LINE__);                                    \
      return DECOMOE_ERR_CUDA;                                                     \
    }                                                                              \
  } while (0)

#define DM_LAUNCH_CHECK(name)                                                      \
  do {                                                                             \
    cudaError_t e_ = cudaGetLastError();                                           \
    if (e_ != cudaSuccess) {                                                       \
      ::decomoe::set_error("launch of %s failed: %s", name, cudaGetErrorString(e_)); \
      return DECOMOE_ERR_CUDA;                                                     \
    }                                                                              \
  } while (0)

#define DM_RET(expr)                 \
  do {                               \
    int r_ = (expr);                 \
    if (r_ != DECOMOE_OK) return r_; \
  } while (0)

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }
inline size_t dtype_bytes(int dtype) { return dtype == DECOMOE_BF16 ? 2 : 4; }

int sm_count();  // cached per device
bool pdl_enabled(int64_t blocks);  // programmatic dependent launch for a grid of this many blocks

// Launch with programmatic stream serialisation: the kernel's CTAs may start
// while the previous kernel on the stream is still running; every kernel
// launched this way calls pdl_wait() before it reads anything an earlier
// kernel wrote (or writes anything an earlier kernel reads).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed =
      pdl_enabled(static_cast<int64_t>(grid.x) * grid.y * grid.z) ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// Internal entry points shared between translation units.
// TMA map of a 2-D bf16 tensor [outer, inner] row-major; box = box_outer rows x
// box_inner columns (64 -> 128-byte swizzle, 32 -> 64-byte swizzle), zero fill
// out of bounds.
int make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint32_t box_outer,
                   uint32_t box_inner);
// 3-D bf16 tensor (dims[0] contiguous; byte strides of dims 1 and 2), box[0]
// = 64 elements with 128-byte swizzle, zero fill out of bounds.
int make_tmap_bf16_3d(CUtensorMap* m, const void* base, const uint64_t dims[3], const uint64_t strides[2],
                      const uint32_t box[3]);
int launch_router_tc(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E,
                     float* logits, int32_t* status, cudaStream_t s);
bool router_tc_supported(int d, int E);
int router_split_ks(int64_t T, int d, int E);  // k slices of the split router at T tokens (1: no split)
int launch_router_split(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E, float* logits,
                        float* scratch, int32_t* status, cudaStream_t s);
int launch_skip_mass(const float* logits, int64_t n, int E, int64_t ld, int k, int64_t skip_at, int64_t skip_len,
                     double* part, double* mass, cudaStream_t s);

// Where the routing kernel reads its logits: row t is
// parts[t*ld + e] + parts[part_stride + t*ld + e] + ... (nparts slices, in
// slice order) + bias[e] (when bias is set), the sum the k-split router's
// reduction forms, so routing can read the router's partial sums directly;
// logits_out (optional) receives the summed rows. Plain logits: nparts = 1,
// no bias, no logits_out.
struct RouteSrc {
  int nparts = 1;
  int64_t part_stride = 0;
  const float* bias = nullptr;
  float* logits_out = nullptr;
};
// Tokens per routing block (one warp per token): up to this many tokens the
// routing launch is a single block.
constexpr int ROUTE_TOKENS_PER_BLOCK = 8;
// Dispatch done by a single routing block right after it has routed its
// tokens (T <= 8): the arguments of decomoe_dispatch for Kd groups, x_perm
// null when the rows are copied by a separate launch. counts null: none.
struct RouteDispatch {
  int32_t* counts = nullptr;
  int32_t* offsets = nullptr;
  int32_t* perm_token = nullptr;
  int32_t* inv_slot = nullptr;
  int32_t* status = nullptr;
  const void* x = nullptr;
  int row_vec = 0;  // 16-byte vectors per row
  void* x_perm = nullptr;
  int Kd = 0;
};
// decomoe_route_prefix reading its logits through src. defer_finalize: with
// mass_out and more than one routing block, the per-block partial masses are
// left in the workspace (their count returned in *mass_blocks) for a later
// kernel to add up (launch_dispatch's extra blocks) instead of a separate
// finalize launch. K_dev: the prefix is read on the device (no mass).
// rd: with one routing block, that block also dispatches its picks.
// zero_ints: n_zero int32 that the launch clears (for a later launch of the
// same chain).
int route_prefix_src(const float* logits, const RouteSrc& src, int64_t T, int E, int64_t ld, int K, int k,
                     int32_t* topk_idx, float* topk_w, double* mass_out, void* ws, size_t ws_bytes,
                     bool defer_finalize, int* mass_blocks, cudaStream_t s, const int32_t* K_dev = nullptr,
                     const RouteDispatch* rd = nullptr, int32_t* zero_ints = nullptr, int n_zero = 0);
// The row gather of decomoe_dispatch: x_perm[r] = x[perm_token[r]] for the
// offsets[K] routed rows (N = T*k rows at most).
int launch_gather_rows(const void* x, const int32_t* perm_token, const int32_t* offsets, int K, size_t row_bytes,
                       int64_t N, void* x_perm, cudaStream_t s);
// decomoe_dispatch that also finishes a deferred activated mass: mass[e] =
// fixed-order fp64 sum of mass_part[b][e] over mass_blocks blocks (no-op when
// mass_part is null).
int dispatch_with_mass(const int32_t* topk_idx, int64_t T, int k, int K, const void* x, int d, int dtype,
                       int32_t* counts, int32_t* offsets, int32_t* perm_token, int32_t* inv_slot, void* x_perm,
                       void* ws, size_t ws_bytes, int32_t* status_dev, const double* mass_part, int mass_blocks,
                       int mass_E, double* mass, cudaStream_t s);
// decomoe_combine, and with text_out also the visual-block removal of its
// output rows (decomoe_combine_drop_visual_block).
int combine_impl(const void* y_perm, const int32_t* inv_slot, const float* topk_w, int64_t T, int k, int d,
                 int dtype, const void* residual, void* out, void* text_out, int64_t v0, int64_t nv,
                 decomoe_stream_t stream, bool discard_y = false);
// Whether calls that own scratch rows drop them from L2 after their last read
// (decomoe_set_discard_scratch; on by default).
bool discard_scratch();
// decomoe_drop_visual_block; with flag, only when *flag == 1 on the device.
int drop_visual_block_impl(const int32_t* flag, const void* src, void* dst, int64_t rows, int64_t row_bytes,
                           int64_t v0, int64_t nv, int64_t nbatch, int64_t src_batch_stride,
                           int64_t dst_batch_stride, decomoe_stream_t stream);
// decomoe_moe_layer; with text_out also the visual-block removal of its output
// (decomoe_moe_layer_exit).
int moe_layer_impl(const void* x, const void* w_r, const float* bias, const void* w_gate_up, const void* w_down,
                   int64_t T, int d, int E, int k, int m, int dtype, int K_fixed, double p, const void* residual,
                   void* out, void* text_out, int64_t v0, int64_t nv, int* K_used_host, int* K_sel_host, void* ws,
                   size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream);
// Both expert GEMMs in one launch (bf16): ready holds
// expert_ffn_sync_ints(rows, K) int32, zero at launch. Sets *launched = false
// (and launches nothing) where the two-launch form is kept. With gather_x and
// perm (tokens-as-M form only) the launch also fills x_perm[r] =
// gather_x[perm[r]] itself.
enum { FFN_FUSED_NONE = 0, FFN_FUSED_WS = 1, FFN_FUSED_TC = 2 };
int expert_ffn_fused_kind(int64_t rows, int K, int m, int dtype);
size_t expert_ffn_sync_ints(int64_t rows, int E);
int launch_expert_ffn_fused(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d, int m, int dtype,
                            const void* w_gate_up, const void* w_down, void* h, void* y_perm, int32_t* ready,
                            int32_t* status, cudaStream_t s, bool* launched, const void* gather_x = nullptr,
                            const int32_t* perm = nullptr);
// One launch for a whole decode-size layer (router, routing, dispatch,
// experts, combine, and with text_out the visual-block removal of the
// output; fixed or device-selected prefix). sync: decode_layer_sync_ints(T, d, E) int32 of the caller's
// workspace, 16-byte aligned, any content (the launch clears what it uses).
bool decode_layer_supported(int64_t T, int d, int E, int k, int m, int dtype, int K_fixed);
size_t decode_layer_sync_ints(int64_t T, int d, int E);
int launch_decode_layer(const void* x, const void* w_r, const float* bias, const void* w_gate_up, const void* w_down,
                        int64_t T, int d, int E, int k, int m, int K_fixed, double p, const void* residual, void* out,
                        void* text_out, int64_t v0, int64_t nv, float* logits, int32_t* topk_idx, float* topk_w, double* mass, int32_t* counts,
                        int32_t* offsets, int32_t* perm, int32_t* inv, void* x_perm, void* h, void* y, int32_t* K_dev,
                        int32_t* sync, int32_t* status, cudaStream_t s);
// The k-split router's GEMM alone: KS slices of partial logits [KS][T][E]
// (no bias) into scratch; returns KS (1: no split at this size, nothing
// launched).
int launch_router_parts(const void* x, const void* w_r, int64_t T, int d, int E, float* scratch, int32_t* status,
                        cudaStream_t s, int* ks_out);

// ---------------------------------------------------------------- device side

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Activated mass of expert e (Eq. 11) from the routing blocks' partial sums,
// by one block of 256 threads: thread i adds blocks i, i + 256, ... in order,
// then a fixed-shape tree combines the 256 thread sums (bit-reproducible, the
// same order wherever it runs).
__device__ __forceinline__ void mass_finalize_block(const double* __restrict__ part, int nblocks, int E, int e,
                                                    double* __restrict__ mass) {
  __shared__ double red[256];
  double acc = 0.0;
  for (int b = threadIdx.x; b < nblocks; b += 256) acc += part[static_cast<int64_t>(b) * E + e];
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) mass[e] = red[0];
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Programmatic dependent launch: let the next kernel on the stream be
// scheduled now, and wait until the previous kernel has completed and its
// memory is visible (a no-op for kernels launched without the attribute).
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_enter() {
  pdl_trigger();
  pdl_wait();
}

// Record the first error code in the caller's status word (if given).
__device__ __forceinline__ void report_status(int32_t* status, int32_t code) {
  if (status != nullptr) atomicCAS(status, 0, code);
}

// Barrier over a subset of the block's warps (named barrier id, thread count).
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
// Order this thread's generic-proxy global writes before later async-proxy
// (TMA) accesses of the same memory.
__device__ __forceinline__ void fence_proxy_async_all() { asm volatile("fence.proxy.async;" ::: "memory"); }
__device__ __forceinline__ int ld_acquire_gpu(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// ---- cp.async (16-byte copies into shared memory, completion on an mbarrier)
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
// Arrive on the mbarrier once every earlier cp.async of this thread has
// landed (the arrival is part of the barrier's expected count).
__device__ __forceinline__ void cp_async_mbar_arrive_noinc(uint32_t bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
// Make shared-memory writes of the generic proxy (cp.async, st.shared)
// visible to the async proxy (tcgen05.mma operand reads).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---- mbarrier
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait until the phase with the given parity has completed, for at most
// limit_ns, or until another role of the CTA has raised *abort. Returns false
// on timeout or abort; never spins without bound.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns,
                                          volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

// ---- TMA (bulk tensor copies global -> shared, completion on an mbarrier)
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* m) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* m, uint32_t bar,
                                            int32_t x, int32_t y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* m, uint32_t bar, int32_t x, int32_t y,
                                            int32_t z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}
// Four rows (row0..row3, any order) of a 2-D tensor whose map has a
// one-row box, columns [col, col + box width), into consecutive rows at dst.
__device__ __forceinline__ void tma_gather4(uint32_t dst, const CUtensorMap* m, uint32_t bar, int32_t col,
                                            int32_t r0, int32_t r1, int32_t r2, int32_t r3) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(col), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const CUtensorMap* m, uint32_t bar,
                                                 int32_t x, int32_t y, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// ---- tcgen05 / TMEM
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D(tmem) (+)= A(smem desc) * B(smem desc)^T, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive (once) on an mbarrier when all prior tcgen05 ops of this thread completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}
__device__ __forceinline__ void tc_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 32 lanes x 32 consecutive fp32 columns: thread i of the warp receives lane
// (base lane + i), columns [col, col + 32).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

// Shared-memory matrix descriptor of a K-major bf16 tile written by TMA with
// a 128-byte (BK = 64 elements) or 64-byte (BK = 32) swizzle: one row of BK
// elements per 128 / 64 bytes, 8-row swizzle atoms 1024 / 512 bytes apart.
// Bits: [0,14) start address >> 4, [16,30) leading byte offset >> 4 (unused
// for swizzled K-major, set to 1), [32,46) stride byte offset >> 4 (the atom
// size), [46,48) descriptor version 1, [49,52) base offset 0, [61,64) layout
// (2 = 128-byte swizzle, 4 = 64-byte swizzle). Tiles start on an atom-aligned
// boundary (1024 bytes here). Advancing K by 16 elements adds 32 bytes.
template <int BK>
__device__ __forceinline__ uint64_t smem_desc_kmajor(uint32_t saddr) {
  static_assert(BK == 64 || BK == 32, "BK must be 64 or 32");
  constexpr uint64_t kSbo = BK == 64 ? 1024 : 512;
  constexpr uint64_t kLayout = BK == 64 ? 2 : 4;
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(1) << 16;
  d |= (kSbo >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= kLayout << 61;
  return d;
}

// Instruction descriptor of tcgen05.mma kind::f16: bf16 x bf16 -> fp32, both
// operands K-major, shape M x N (M in {64,128}, N % 16 == 0, N <= 256).
// Bits: [4,6) D format (1 = f32), [7,10) A format (1 = bf16), [10,13) B format
// (1 = bf16), 15/16 A/B major (0 = K), [17,23) N >> 3, [24,29) M >> 4.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// silu(z) = z * sigmoid(z) with the fast exponential and division intrinsics
// (a few ulp in fp32; the results are rounded to bf16).
__device__ __forceinline__ float silu_f(float z) { return __fdividef(z, 1.0f + __expf(-z)); }

}  // namespace decomoe
