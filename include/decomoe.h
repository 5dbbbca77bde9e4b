/*
 * decomoe.h - C ABI of the DecoMoE prefix-MoE hot path on one GB300 (sm_103a).
 *
 * The DecoMoE paper ("DecoMoE: Decoupling Visual Propagation and Expert
 * Computation for Efficient Multimodal MoE Inference") restricts each MoE
 * layer after the visual exit to the shortest contiguous prefix [0, K) of
 * offline mass-reordered experts (RCEP, Section 3.3, Eqs. 10-12, Algorithm 2)
 * and removes the contiguous visual-token block from the hidden state and the
 * KV cache at the exit layer (SAVB, Section 3.2). This library computes the
 * per-layer steps of that path with hand-written CUDA kernels.
 *
 * Conventions (every call):
 *   - extern "C"; every call returns an int status (decomoe_status). No
 *     exception crosses the ABI. On an error the message of the calling host
 *     thread is available from decomoe_last_error().
 *   - The caller owns all memory. Pointers named *_host are host pointers; all
 *     others are device pointers of the current CUDA device. The library never
 *     allocates device memory: temporary space comes from a caller-provided
 *     workspace whose size a *_workspace_bytes() query returns.
 *   - Device calls are asynchronous on the given stream (NULL = legacy default
 *     stream). Outputs are valid after the stream is synchronised; inputs must
 *     stay alive until then. Calls that must read a device value on the host
 *     (decomoe_moe_layer in mass mode, decomoe_read_status) synchronise the
 *     stream and say so.
 *   - Index arrays are int32, row-major. T = tokens of the invocation, d =
 *     hidden size, E = experts in the pool, K = prefix length, k = top-k width,
 *     m = expert FFN width.
 *   - Argument errors (null pointer, k > K, K > E, negative sizes, d or m not a
 *     multiple of the required granule, misaligned pointer) return
 *     DECOMOE_ERR_INVALID_ARG before anything is launched.
 */
#ifndef DECOMOE_H
#define DECOMOE_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define DECOMOE_API __attribute__((visibility("default")))
#else
#define DECOMOE_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* decomoe_stream_t; /* same type as cudaStream_t */

typedef enum {
  DECOMOE_OK = 0,
  DECOMOE_ERR_INVALID_ARG = 1, /* bad argument; nothing was launched */
  DECOMOE_ERR_CUDA = 2,        /* a CUDA launch or API error; see decomoe_last_error() */
  DECOMOE_ERR_TIMEOUT = 3,     /* a bounded device-side wait ran out (read via decomoe_read_status) */
  DECOMOE_ERR_UNSUPPORTED = 4, /* a shape or dtype no kernel here takes */
  DECOMOE_ERR_WORKSPACE = 5,   /* workspace pointer null or smaller than the query says */
  DECOMOE_ERR_BAD_INPUT = 6    /* device-side input check failed (e.g. expert id >= K) */
} decomoe_status;

/* Storage dtype of activations and weights. Accumulation is always fp32 (fp64
 * for the activated mass). */
enum { DECOMOE_BF16 = 0, DECOMOE_F32 = 1 };

/* Gate/up interleave granule of the fused weight layout (rows of one block). */
#define DECOMOE_GU_BLOCK 64
/* Largest expert pool and largest top-k any kernel here takes. */
#define DECOMOE_MAX_E 256
#define DECOMOE_MAX_TOPK 32

/* Message of the last failed call made by this host thread ("" if none). */
DECOMOE_API const char* decomoe_last_error(void);

/* Library ABI version (major*100 + minor). */
DECOMOE_API int decomoe_version(void);

/* Number of SMs and compute capability of the current device. */
DECOMOE_API int decomoe_device_info(int* sm_count_host, int* cc_major_host, int* cc_minor_host);

/* ------------------------------------------------------------------------
 * a1. Router logits over the whole pool (Section 3.1, Eq. 1; the full-pool
 * router projection stays in every layer, Appendix FLOPs "Scope").
 *   logits[t, e] = sum_j x[t, j] * w_r[e, j] + bias[e]      (fp32 out)
 * x: [T, d] row-major, dtype; w_r: [E, d] row-major, dtype, rows in reordered
 * expert order; bias: [E] fp32 or NULL; logits: [T, E] fp32 row-major.
 * bf16 with T <= 6 and d % 8 == 0 runs a CUDA-core dot-product kernel (one
 * block per router row); above that, d % 64 == 0 and E in {128, 256} run on
 * the tensor cores (fp32 accumulate); f32 and other bf16 shapes run a
 * CUDA-core kernel.
 * status_dev: optional device int32 that collects bounded-wait timeouts.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_router_logits(const void* x, const void* w_r, const float* bias, int64_t T, int d,
                          int E, int dtype, float* logits, int32_t* status_dev,
                          decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a1 with a workspace: the same logits as decomoe_router_logits (within the
 * fp32 summation bound; the order of the additions differs). Above the
 * CUDA-core token range the tensor-core router then splits the k loop into
 * slices that run on more CTAs and adds their partial sums in slice order,
 * the bias last. ws: decomoe_router_logits_ws_bytes(T, d, E) bytes (0 means
 * no split at this size; ws may then be NULL), 16-byte aligned.
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_router_logits_ws_bytes(int64_t T, int d, int E);
DECOMOE_API int decomoe_router_logits_ws(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E,
                                         int dtype, float* logits, void* ws, size_t ws_bytes, int32_t* status_dev,
                                         decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a2 + a4. Routing on fp32 logits (Eqs. 10-11; prefix rule of Section 3.3 and
 * Algorithm 2).
 *   For every token t: S_t = the k largest of logits[t, 0:K) (largest first;
 *   equal values: lower expert index first), and
 *   topk_w[t, j] = exp(l_j - l_0) / sum_j' exp(l_j' - l_0) over the k picks,
 *   which equals "new softmax over the prefix, top-k, renormalise".
 *   With K == E this is the full-pool routing of Eq. 10. If mass_out is not
 *   NULL the same launch also computes the activated mass of Eq. 11 over the
 *   full pool [0, E) whatever K is: mass_out[e] = sum over tokens of the
 *   renormalised full-pool top-k weight of e (fp32 weights, fp64 sum across
 *   blocks in a fixed order: bit-reproducible run to run, relative error of a
 *   few 1e-7); mass_out then needs E entries and the workspace.
 * logits: [T, ld] fp32, entries [0, E) used, ld >= E. topk_idx: [T, k] int32,
 * values in [0, K). topk_w: [T, k] fp32. Either output may be NULL (e.g. the
 * mass-only pass). Needs 1 <= k <= K <= E <= 256, k <= 32.
 * ws: device workspace of decomoe_route_workspace_bytes(T, E) bytes (only when
 * mass_out != NULL).
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_route_workspace_bytes(int64_t T, int E);
DECOMOE_API int decomoe_route_prefix(const float* logits, int64_t T, int E, int64_t ld, int K, int k,
                         int32_t* topk_idx, float* topk_w, double* mass_out, void* ws,
                         size_t ws_bytes, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a3. Prefix length (Eq. 12), plain C on the host, no CUDA.
 *   K_hat = min{K in 1..E : sum_{e<K} mass[e] / sum_e mass[e] >= p},
 *   K = max(k, K_hat). Sums run sequentially over e = 0..E-1 in fp64; p == 1
 *   gives K_hat = E; a total mass of 0 gives K = k.
 * mass_host: [E] fp64 host array. Needs 0 < p <= 1, 1 <= k <= E.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_select_prefix(const double* mass_host, int E, int k, double p, int* K_out_host);

/* ------------------------------------------------------------------------
 * Prefix selection on the device (Eq. 12 as decomoe_select_prefix, same
 * sequential fp64 arithmetic, so the same K bit for bit): reads mass [E]
 * (e.g. the mass_out of decomoe_route_prefix) and writes K to K_dev (one
 * int32 on the device). With decomoe_route_prefix_dk, which routes over the
 * prefix [0, *K_dev), the mass-selected RCEP layer needs no host
 * synchronisation: dispatch and the expert GEMMs then take K = E (experts at
 * or beyond *K_dev receive no rows and cost nothing).
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_select_prefix_device(const double* mass, int E, int k, double p, int32_t* K_dev,
                                             decomoe_stream_t stream);
DECOMOE_API int decomoe_route_prefix_dk(const float* logits, int64_t T, int E, int64_t ld, const int32_t* K_dev,
                                        int k, int32_t* topk_idx, float* topk_w, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a5. Dispatch: group the T*k (token, slot) pairs by expert (Algorithm 2,
 * "evaluate ... only the first K expert MLPs").
 *   counts[e] = #pairs with topk_idx == e (e < K); offsets = exclusive scan,
 *   offsets[K] = T*k. Rows are ordered by expert, then by flat index
 *   f = t*k + j (a stable sort). perm_token[r] = token of row r;
 *   inv_slot[f] = row of pair f; x_perm[r, :] = x[perm_token[r], :].
 * topk_idx: [T, k] int32 in [0, K) (an id outside it sets DECOMOE_ERR_BAD_INPUT
 * in status_dev, if given, and that pair is dropped). x: [T, d] dtype (rows
 * 16-byte aligned); x_perm: [T*k, d] dtype, or NULL to skip the row gather.
 * counts: [K], offsets: [K+1], perm_token and inv_slot: [T*k] int32.
 * ws: decomoe_dispatch_workspace_bytes(T, k, K) bytes.
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_dispatch_workspace_bytes(int64_t T, int k, int K);
/* The row gather of the dispatch alone: x_perm[r, :] = x[perm_token[r], :]
 * for the offsets[K] (<= N) rows counted on the device (from a dispatch run
 * without x_perm). x: [T, d] dtype, x_perm: [N, d] dtype, both 16-byte
 * aligned with rows of a multiple of 16 bytes (DECOMOE_ERR_INVALID_ARG
 * otherwise). */
DECOMOE_API int decomoe_gather_rows(const void* x, const int32_t* perm_token, const int32_t* offsets, int K,
                                    int64_t N, int d, int dtype, void* x_perm, decomoe_stream_t stream);
DECOMOE_API int decomoe_dispatch(const int32_t* topk_idx, int64_t T, int k, int K, const void* x, int d,
                     int dtype, int32_t* counts, int32_t* offsets, int32_t* perm_token,
                     int32_t* inv_slot, void* x_perm, void* ws, size_t ws_bytes,
                     int32_t* status_dev, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a2-a5 in one call: routing and dispatch of one RCEP invocation (Eqs.
 * 10-12 and the prefix routing and dispatch of Algorithm 2). Outputs are
 * bit-identical to decomoe_route_prefix (+ decomoe_select_prefix_device +
 * decomoe_route_prefix_dk) followed by decomoe_dispatch on the same logits.
 *   K >= k (<= E): fixed prefix [0, K); with mass_out ([E] fp64) the call also
 *     computes the full-pool activated mass of Eq. 11; p is ignored.
 *     Dispatch groups: K.
 *   K == -1: device-selected prefix: mass_out (required) gets the mass, K is
 *     chosen by Eq. 12 with 0 < p <= 1 (decomoe_select_prefix's arithmetic)
 *     and written to K_dev (required), routing runs over [0, K). Dispatch
 *     groups: E (those at or beyond K stay empty): counts [E], offsets [E+1].
 * logits: [T, E] fp32 (row stride E). topk_idx, topk_w: [T, k]. x, d, dtype,
 * counts, offsets, perm_token, inv_slot, x_perm: as decomoe_dispatch (x_perm
 * NULL skips the row gather).
 * ws: decomoe_route_dispatch_workspace_bytes(T, k, E) bytes (the routing
 * and dispatch scratch). No host synchronisation; capturable in a CUDA graph.
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_route_dispatch_workspace_bytes(int64_t T, int k, int E);
DECOMOE_API int decomoe_route_dispatch(const float* logits, int64_t T, int E, int K, int k, double p,
                                       int32_t* topk_idx, float* topk_w, double* mass_out, int32_t* K_dev,
                                       const void* x, int d, int dtype, int32_t* counts, int32_t* offsets,
                                       int32_t* perm_token, int32_t* inv_slot, void* x_perm, void* ws,
                                       size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a1-a5 in one call: the router logits over the full pool (Eq. 10's input),
 * then decomoe_route_dispatch on them. Outputs (logits included) are
 * bit-identical to decomoe_router_logits_ws followed by
 * decomoe_route_dispatch with the same arguments. Where the router splits
 * its k loop (bf16, 6 < T, k slices that fit the SMs), the routing kernel
 * reads the router's partial sums itself, adding them in slice order and the
 * bias last exactly as the router's own reduction does, and writes the summed
 * logits; with a fixed K and mass_out the activated mass is added up by the
 * dispatch launch. Two launches fewer than the separate calls.
 * x: [T, d] dtype; w_r: [E, d] dtype; bias: [E] fp32 or NULL; logits: [T, E]
 * fp32 output (required). K, k, p, topk_idx, topk_w, mass_out, K_dev,
 * counts, offsets, perm_token, inv_slot, x_perm: as decomoe_route_dispatch
 * (x, d and dtype are the dispatch's too).
 * ws: decomoe_router_route_dispatch_workspace_bytes(T, d, E, k) bytes, 16-byte
 * aligned (the split router's partials, then the routing and dispatch
 * scratch). No host synchronisation; capturable in a CUDA graph.
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_router_route_dispatch_workspace_bytes(int64_t T, int d, int E, int k);
DECOMOE_API int decomoe_router_route_dispatch(const void* x, const void* w_r, const float* bias, int64_t T,
                                              int d, int E, int dtype, int K, int k, double p, float* logits,
                                              int32_t* topk_idx, float* topk_w, double* mass_out,
                                              int32_t* K_dev, int32_t* counts, int32_t* offsets,
                                              int32_t* perm_token, int32_t* inv_slot, void* x_perm, void* ws,
                                              size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Allocation-free dispatch (the paper has no counterpart: this is a library
 * convenience). Same arguments, outputs and errors as decomoe_dispatch, minus
 * the workspace: for callers that cannot allocate device memory, e.g. a
 * serving runtime that owns all of HBM in a fixed arena from start-up and
 * forbids later cudaMalloc (it can synchronise the device and fragment the
 * arena). The per-tile histograms then live in a fixed array inside the
 * library image, of DECOMOE_NOALLOC_DISPATCH_SCRATCH_INTS int32 entries
 * (256 KiB), which every GPU that loads the library keeps until the process
 * exits. Requires ceil(T*k / 1024) * K <= that size, else
 * DECOMOE_ERR_INVALID_ARG with a message and nothing launched.
 *   - The first call on a device looks up the array's device address (once
 *     per device, with that device current); make that first call before any
 *     stream capture. A first call made while its stream is capturing returns
 *     DECOMOE_ERR_INVALID_ARG and launches nothing.
 *   - The address is cached per device ordinal for the life of the process:
 *     it assumes the device's primary context outlives every call and is not
 *     looked up again after cudaDeviceReset.
 *   - Calls never allocate or free device memory.
 *   - All calls on a device share the one array and it keeps the last call's
 *     contents; nothing in it needs to start at zero (each call writes every
 *     entry it reads). Calls whose execution overlaps on the GPU (different
 *     streams, or other threads) race on the array: serialise them.
 * ------------------------------------------------------------------------ */
#define DECOMOE_NOALLOC_DISPATCH_SCRATCH_INTS 65536
DECOMOE_API int decomoe_dispatch_noalloc(const int32_t* topk_idx, int64_t T, int k, int K, const void* x,
                                         int d, int dtype, int32_t* counts, int32_t* offsets,
                                         int32_t* perm_token, int32_t* inv_slot, void* x_perm,
                                         int32_t* status_dev, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * One-time weight layout transform (like the paper's load-time expert
 * reorder, Section 3.3: it changes storage only, not values).
 *   w_gate, w_up: [E, m, d] row-major (dtype). w_gate_up: [E, 2m, d], where
 *   rows [2*G*b, 2*G*b + G) of expert e are gate rows [G*b, G*b + G) and rows
 *   [2*G*b + G, 2*G*(b+1)) are up rows [G*b, G*b + G), G = DECOMOE_GU_BLOCK.
 * Needs m % 128 == 0.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_weight_layout(const void* w_gate, const void* w_up, void* w_gate_up, int E, int d,
                          int m, int dtype, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a6. Grouped SwiGLU expert FFN over the prefix experts (Algorithm 2; gate,
 * up and down matmuls, Appendix C_expert = 6Kdm).
 *   For every row r in [offsets[e], offsets[e+1]), e < K:
 *   h_r = silu(W_gate[e] x_r) * (W_up[e] x_r); y_r = W_down[e] h_r.
 * x_perm: [rows, d]; w_gate_up: [E, 2m, d] in the layout above; w_down:
 * [E, d, m]; h_ws: [rows, m] dtype (intermediate, caller-owned); y_perm:
 * [rows, d] dtype. rows = T*k = offsets[K] (upper bound used to size tensor
 * maps; offsets stay on the device). Experts with no rows cost nothing.
 * bf16: tcgen05 tensor-core kernels for rows > 64, a weight-streaming kernel
 * for rows <= 64 (decode); fp32 accumulate, h rounded to bf16. f32: CUDA-core
 * kernels with h kept in fp32. Needs m % 64 == 0; bf16 also m % 128 == 0,
 * d % 256 == 0 and 16-byte aligned pointers (DECOMOE_ERR_INVALID_ARG
 * otherwise, before any launch).
 * status_dev: optional device int32 collecting bounded-wait timeouts.
 * sched_dev: optional device int32 (4 bytes, caller-owned). Given, the
 * tensor-core kernels hand tiles out dynamically from this counter (the call
 * zeroes it first) instead of a fixed round robin, which balances the mix of
 * weight-streaming and weight-reusing tiles. Launches that may overlap on the
 * GPU need distinct counters. NULL keeps the static order.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_expert_swiglu(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d,
                          int m, int dtype, const void* w_gate_up, const void* w_down, void* h_ws,
                          void* y_perm, int32_t* status_dev, int32_t* sched_dev, decomoe_stream_t stream);

/* decomoe_expert_swiglu with both GEMMs in one persistent launch where that
 * is faster (bf16, 16 to 32768 rows): the down tiles of an expert (decode
 * sizes) or of a 128-row tile (larger) start as soon as the gate/up tiles
 * they read have stored h, published through per-expert or per-tile counters
 * with release/acquire ordering. ready: decomoe_expert_swiglu_ready_ints(rows,
 * K) int32, all zero at the call (decomoe_moe_layer clears its own); the call
 * leaves them non-zero. Outside that range the call runs the two launches of
 * decomoe_expert_swiglu and leaves ready untouched. Outputs are bit-identical
 * to decomoe_expert_swiglu. Needs every CTA of the launch resident at once
 * (it sizes the grid to the SMs of the current device). */
DECOMOE_API size_t decomoe_expert_swiglu_ready_ints(int64_t rows, int K);
DECOMOE_API int decomoe_expert_swiglu_fused(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d,
                                            int m, int dtype, const void* w_gate_up, const void* w_down, void* h_ws,
                                            void* y_perm, int32_t* ready, int32_t* status_dev,
                                            decomoe_stream_t stream);

/* The same one launch as decomoe_moe_layer runs it from 8192 routed rows: the
 * dispatch's row gather inside the expert launch (Algorithm 2, dispatch and
 * expert evaluation). x: [T, d] token rows; perm_token: [rows] from
 * decomoe_dispatch (called without x_perm); x_perm: [rows, d] scratch the
 * launch fills with x[perm_token[r]] on its way to the tiles (caller-owned,
 * 16-byte aligned). Other arguments as decomoe_expert_swiglu_fused; ready
 * needs decomoe_expert_swiglu_ready_ints(rows, K) zeroed int32. Only for
 * sizes the one-launch tokens-as-M form takes (bf16, 8*K < rows <= 32768):
 * DECOMOE_ERR_INVALID_ARG otherwise, nothing launched. Outputs equal those of
 * decomoe_dispatch with x_perm followed by decomoe_expert_swiglu, bit for bit. */
DECOMOE_API int decomoe_expert_swiglu_fused_gather(const void* x, int64_t T, const int32_t* perm_token,
                                                   const int32_t* offsets, int64_t rows, int K, int d, int m,
                                                   int dtype, const void* w_gate_up, const void* w_down,
                                                   void* x_perm, void* h_ws, void* y_perm, int32_t* ready,
                                                   int32_t* status_dev, decomoe_stream_t stream);

/* The two phases of decomoe_expert_swiglu as separate calls (same arguments
 * and rules): gate/up with the fused SwiGLU epilogue writes h [rows, m]; down
 * reads h and writes y_perm [rows, d]. */
DECOMOE_API int decomoe_expert_gate_up(const void* x_perm, const int32_t* offsets, int64_t rows, int K, int d,
                                       int m, int dtype, const void* w_gate_up, void* h, int32_t* status_dev,
                                       int32_t* sched_dev, decomoe_stream_t stream);
DECOMOE_API int decomoe_expert_down(const void* h, const int32_t* offsets, int64_t rows, int K, int d, int m,
                                    int dtype, const void* w_down, void* y_perm, int32_t* status_dev,
                                    int32_t* sched_dev, decomoe_stream_t stream);

/* Gather forms: the expert rows are read straight from the token-ordered
 * hidden state, row r of the grouped order being x[perm_token[r], :] (TMA
 * tile::gather4 on the tensor cores), so dispatch need not materialise x_perm
 * (saves T*k*d elements of memory). Same results bit for bit as the x_perm
 * forms; slower at prefill sizes, where the four-row gathers, not the tensor
 * cores, bound the gate/up GEMM. x: [T, d] dtype; perm_token: [rows] int32
 * from decomoe_dispatch; other arguments and rules as decomoe_expert_gate_up /
 * decomoe_expert_swiglu. */
DECOMOE_API int decomoe_expert_gate_up_gather(const void* x, int64_t T, const int32_t* perm_token,
                                              const int32_t* offsets, int64_t rows, int K, int d, int m,
                                              int dtype, const void* w_gate_up, void* h, int32_t* status_dev,
                                              int32_t* sched_dev, decomoe_stream_t stream);
DECOMOE_API int decomoe_expert_swiglu_gather(const void* x, int64_t T, const int32_t* perm_token,
                                             const int32_t* offsets, int64_t rows, int K, int d, int m, int dtype,
                                             const void* w_gate_up, const void* w_down, void* h_ws,
                                             void* y_perm, int32_t* status_dev, int32_t* sched_dev,
                                             decomoe_stream_t stream);

/* CUDA-core reference of decomoe_expert_swiglu for bf16 storage: the same
 * arithmetic (bf16 products, fp32 accumulation, h rounded to bf16) with one
 * thread per output element and no tensor cores. It is slow; it exists to
 * localise a disagreement between the tensor-core kernels and the oracle. */
DECOMOE_API int decomoe_expert_swiglu_ref(const void* x_perm, const int32_t* offsets, int64_t rows, int K,
                                          int d, int m, const void* w_gate_up, const void* w_down,
                                          void* h_ws, void* y_perm, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a7. Combine (Algorithm 2, "evaluate and combine"): the weighted sum of a
 * token's k expert outputs, written as a gather (deterministic, no atomics).
 *   out[t, :] = sum_{j=0..k-1} topk_w[t, j] * y_perm[inv_slot[t*k + j], :]
 *               (+ residual[t, :])
 * fp32 sum in slot order j = 0..k-1, rounded once to dtype. residual may be
 * NULL. out must not alias y_perm.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_combine(const void* y_perm, const int32_t* inv_slot, const float* topk_w, int64_t T,
                    int k, int d, int dtype, const void* residual, void* out,
                    decomoe_stream_t stream);

/* a7 + a8 in one launch: decomoe_combine, and every text row of its output
 * (t < v0 or t >= v0 + nv, the rows outside the visual block of Section 3.2)
 * also stored to text_out [T - nv, d] in order, the block's rows skipped.
 * out and text_out are bit-identical to decomoe_combine followed by
 * decomoe_drop_visual_block(out, text_out, T, d * elem, v0, nv, 1, ...).
 * Needs 0 <= v0, 0 <= nv, v0 + nv <= T; text_out 16-byte aligned and not
 * overlapping out (else DECOMOE_ERR_INVALID_ARG, nothing launched). */
DECOMOE_API int decomoe_combine_drop_visual_block(const void* y_perm, const int32_t* inv_slot,
                                                  const float* topk_w, int64_t T, int k, int d, int dtype,
                                                  const void* residual, void* out, void* text_out, int64_t v0,
                                                  int64_t nv, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * a8. Visual-block removal (Section 3.2: the complete visual block leaves the
 * hidden state and the KV cache; later layers and decoding use the text-only
 * sequence). Out-of-place, order-preserving row compaction, batched:
 *   for b < nbatch: dst[b] = rows [0, v0) of src[b] followed by rows
 *   [v0 + nv, rows) of src[b].
 * row_bytes: bytes per row; src_batch_stride / dst_batch_stride: bytes between
 * consecutive batches (rows of one batch are contiguous). src and dst must not
 * overlap. 0 <= v0, 0 <= nv, v0 + nv <= rows; nv == 0 is a plain copy.
 * 16-byte aligned pointers, row_bytes and strides take the vector path; any
 * other alignment takes a byte path.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_drop_visual_block(const void* src, void* dst, int64_t rows, int64_t row_bytes,
                              int64_t v0, int64_t nv, int64_t nbatch, int64_t src_batch_stride,
                              int64_t dst_batch_stride, decomoe_stream_t stream);

/* The SAVB trigger fused into the removal (Section 3.2, Eq. 3): the same
 * call with the gate's device-side decision exit_flag (decomoe_savb_gate's
 * exit_flag_dev). The kernel reads *exit_flag: 1 performs the removal above,
 * any other value writes nothing to dst. A caller can queue the removal of
 * the hidden state and of the KV slices right behind the gate and read the
 * decision back afterwards, instead of between the gate and the removal.
 * Arguments and errors as decomoe_drop_visual_block; exit_flag must not be
 * NULL (DECOMOE_ERR_INVALID_ARG). */
DECOMOE_API int decomoe_drop_visual_block_if(const int32_t* exit_flag, const void* src, void* dst, int64_t rows,
                                             int64_t row_bytes, int64_t v0, int64_t nv, int64_t nbatch,
                                             int64_t src_batch_stride, int64_t dst_batch_stride,
                                             decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * SAVB exit gate (Section 3.2, Eqs. 2-3), evaluated at the candidate layers
 * {3, 7, ..., 47} (zero-based, Appendix) on the hidden state h [T, d]:
 *   text rows = rows outside the visual block [v0, v0+nv), in order (n of
 *   them, n >= 1); x = [mean of text rows 0..n-2 ; text row n-1] (fp32 sums
 *   in a fixed order; the pooled half is 0 when n == 1);
 *   z = W2 relu(W1 x + b1) + b2 (hidden width H; ReLU is this library's
 *   reading, the paper does not name the activation);
 *   p_exit = softmax(z)_1, exit = [p_exit >= theta].
 * h: dtype (DECOMOE_BF16 or DECOMOE_F32), d a multiple of 64, 16-byte
 * aligned. w1 [H, 2d], b1 [H], w2 [2, H], b2 [2]: fp32 device arrays (w1
 * 16-byte aligned). p_exit, exit_flag: one fp32 / int32 on the device.
 * ws: decomoe_savb_gate_workspace_bytes(d, H) bytes, 16-byte aligned; it
 * need not start at zero. Two launches; no host synchronisation (the caller
 * reads exit_flag to decide whether to remove the visual block before the
 * next layer, which changes the shapes of every later launch).
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_savb_gate_workspace_bytes(int d, int H);
DECOMOE_API int decomoe_savb_gate(const void* h, int64_t T, int d, int dtype, int64_t v0, int64_t nv,
                                  const float* w1, const float* b1, const float* w2, const float* b2, int H,
                                  float theta, float* p_exit, int32_t* exit_flag, void* ws, size_t ws_bytes,
                                  decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Offline RCEP calibration (Section 3.3, Eqs. 8-9; Algorithm 1).
 *
 * decomoe_calib_case_mass: one calibration case at one layer. logits [T, ld]
 * fp32 are the router logits of the case's sequence; its text tokens are the
 * rows outside the visual block [v0, v0+nv) (n = T - nv >= 1). Adds the
 * case's text-token routed mass of Eq. 9 to accum:
 *   accum[e] += (1/n) * sum over text tokens of the renormalised full-pool
 *               top-k weight of e
 * (the same fp32 weights and fixed-order fp64 sums as the activated mass of
 * decomoe_route_prefix, then one fp64 division; cases add in call order).
 * accum: [E] fp64 on the device, zeroed by the caller before the first case.
 * ws: decomoe_calib_workspace_bytes(T, E) bytes. Needs 1 <= k <= E <= 256.
 *
 * decomoe_mean_mass_order: Eq. 8. mean[e] = accum[e] / n_cases; pi[i] = the
 * expert at new position i, by descending mean, equal means in ascending
 * expert index. pi: [E] int32 on the device; mean_out: [E] fp64 or NULL. A
 * NaN mean sets DECOMOE_ERR_BAD_INPUT in status_dev.
 *
 * decomoe_permute_experts: the one-time reorder of Algorithm 1's last loop:
 * dst expert block i = src expert block pi[i], for a tensor stored as E
 * consecutive blocks of bytes_per_expert bytes (router rows [E, d], the
 * router bias [E], gate/up [E, 2m, d] in either layout, down [E, d, m]).
 * Out of place (src and dst must not overlap). An index outside [0, E) sets
 * DECOMOE_ERR_BAD_INPUT and leaves that block unwritten; pi must be a
 * permutation for dst to hold every expert.
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_calib_workspace_bytes(int64_t T, int E);
DECOMOE_API int decomoe_calib_case_mass(const float* logits, int64_t T, int E, int64_t ld, int k, int64_t v0,
                                        int64_t nv, double* accum, void* ws, size_t ws_bytes,
                                        decomoe_stream_t stream);
DECOMOE_API int decomoe_mean_mass_order(const double* accum, int E, int n_cases, int32_t* pi, double* mean_out,
                                        int32_t* status_dev, decomoe_stream_t stream);
DECOMOE_API int decomoe_permute_experts(const void* src, void* dst, const int32_t* pi, int E,
                                        int64_t bytes_per_expert, int32_t* status_dev, decomoe_stream_t stream);

/* RMSNorm of the attention-free layer stack (a workload choice; the paper
 * leaves norms out of the method): y[t] = x[t] / sqrt(mean(x[t]^2) + eps),
 * fp32 math, dtype in and out. y may alias x. */
DECOMOE_API int decomoe_rmsnorm(const void* x, void* y, int64_t T, int d, float eps, int dtype,
                    decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Whole RCEP MoE invocation (Algorithm 2, exited branch), chaining a1..a7 on
 * one stream:
 *   router logits -> [mass pass -> select prefix] -> prefix routing ->
 *   dispatch -> grouped SwiGLU -> combine (+ residual).
 * K_fixed > 0 routes over the fixed prefix [0, K_fixed) (the paper's fixed
 * keep-ratio experiments); with p > 0 the same routing launch also leaves the
 * full-pool activated mass in the workspace (no host sync). K_fixed == 0
 * selects K from p (0 < p <= 1) on the host: the stream is synchronised once
 * to read the mass and K_used_host / K_sel_host receive K. K_fixed == -1
 * selects K from p on the device (decomoe_select_prefix_device): no host
 * synchronisation, capturable in a CUDA graph; K is left as an int32 in the
 * workspace (entry 11 of decomoe_moe_layer_workspace_layout) and the host
 * outputs are set to -1. p == 0 with K_fixed > 0 skips the mass pass.
 * K_used_host / K_sel_host may be NULL.
 * x, residual, out: [T, d] dtype (out may alias residual, not x).
 * ws: decomoe_moe_layer_workspace_bytes(...) bytes; every intermediate
 * (logits, routes, dispatch arrays, x_perm, h, y_perm) lives there.
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_moe_layer_workspace_bytes(int64_t T, int d, int E, int k, int m, int dtype);
DECOMOE_API int decomoe_moe_layer(const void* x, const void* w_r, const float* bias, const void* w_gate_up,
                      const void* w_down, int64_t T, int d, int E, int k, int m, int dtype,
                      int K_fixed, double p, const void* residual, void* out, int* K_used_host,
                      int* K_sel_host, void* ws, size_t ws_bytes, int32_t* status_dev,
                      decomoe_stream_t stream);

/* The exit layer of Algorithm 2: decomoe_moe_layer whose output also leaves
 * the visual block (Section 3.2) in the same combine launch: out [T, d] as
 * decomoe_moe_layer writes it, and its text rows (outside [v0, v0 + nv)) in
 * order in text_out [T - nv, d] — bit-identical to decomoe_moe_layer followed
 * by decomoe_drop_visual_block(out, text_out, ...). Needs 0 <= v0, 0 <= nv,
 * v0 + nv <= T, text_out 16-byte aligned and apart from out (may be NULL
 * when nv == T). Other arguments as decomoe_moe_layer. */
DECOMOE_API int decomoe_moe_layer_exit(const void* x, const void* w_r, const float* bias, const void* w_gate_up,
                                       const void* w_down, int64_t T, int d, int E, int k, int m, int dtype,
                                       int K_fixed, double p, const void* residual, void* out, void* text_out,
                                       int64_t v0, int64_t nv, int* K_used_host, int* K_sel_host, void* ws,
                                       size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream);

/* Offsets (bytes) of the intermediates inside the decomoe_moe_layer workspace,
 * for inspection: logits, topk_idx, topk_w, mass, counts, offsets, perm_token,
 * inv_slot, x_perm, h, y_perm, device K (12 entries written to offs_host).
 * The layer's scratch rows are dropped from L2 after their last read (see
 * decomoe_set_discard_scratch): turn that off before a call whose y_perm is
 * to be inspected. */
DECOMOE_API int decomoe_moe_layer_workspace_layout(int64_t T, int d, int E, int k, int m, int dtype,
                                       size_t* offs_host);

/* ------------------------------------------------------------------------
 * Attention on the compacted sequence and over the text-only KV cache
 * (Section 3.2: once the visual block exits, attention in that layer and
 * every later one runs on the shortened text-only sequence; Algorithm 2,
 * last step: decoding reuses the shortened cache; Appendix FLOPs 2qS(S+1)
 * per prefill layer, 4qC per decode forward with cache length C).
 *   q: [n, Hq, D] queries of the last n positions; k_cache, v_cache:
 *   [C, Hkv, D] keys and values of the whole (compacted) sequence, the
 *   queries' own rows last (n <= C); out: [n, Hq, D]. All bf16, row-major,
 *   16-byte aligned; D = 128; Hq a multiple of Hkv. Query i sits at position
 *   C - n + i and sees keys 0 .. C - n + i; query head h reads KV head
 *   h / (Hq / Hkv). scale <= 0 means 1 / sqrt(D). fp32 scores, softmax and
 *   accumulation; out rounded to bf16.
 *   Decode sizes: n * (Hq / Hkv) <= 64 queries per KV head: each block
 *   streams a range of keys and keeps the online softmax of up to 32 queries
 *   of its KV head, and the ranges of a thread-block cluster (up to 16
 *   blocks) are merged in key order through the cluster's shared memory. One
 *   cluster per head and no workspace (0 bytes; ws may be null) while that
 *   streams at most four 128-key chunks per block; a longer cache is split
 *   over several clusters per head where the SMs allow, each leaving its
 *   merged rows in the workspace, and a second small launch merges them in
 *   cluster order (deterministic in both cases).
 *   Prefill sizes (more queries per KV head, n = C or a chunk n < C; Hq / Hkv
 *   even): V is transposed into the workspace, then one tensor-core CTA per
 *   (pair of query heads, 128-query tile) runs the online softmax over 64-key
 *   blocks up to its causal limit (P rounded to bf16 before the P V product;
 *   deterministic).
 *   ws: decomoe_attention_workspace_bytes(n, C, Hq, Hkv, D) bytes, 16-byte
 *   aligned. A wait that runs past the time limit records
 *   DECOMOE_ERR_TIMEOUT in status_dev (may be null).
 *   DECOMOE_ERR_INVALID_ARG for other shapes, before any launch.
 * ------------------------------------------------------------------------ */
DECOMOE_API size_t decomoe_attention_workspace_bytes(int64_t n, int64_t C, int Hq, int Hkv, int D);
DECOMOE_API int decomoe_attention(const void* q, int64_t n, const void* k_cache, const void* v_cache, int64_t C,
                                  int Hq, int Hkv, int D, float scale, void* out, void* ws, size_t ws_bytes,
                                  int32_t* status_dev, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Bounded-wait status. Kernels that wait on device barriers give up after a
 * time limit, record DECOMOE_ERR_TIMEOUT (or DECOMOE_ERR_BAD_INPUT) in the
 * caller's status word and return, leaving the context usable.
 * decomoe_read_status synchronises the stream, copies the word to
 * *code_host, clears it and returns DECOMOE_OK.
 * decomoe_set_wait_limit_ns sets the limit used by later launches (default
 * 2e9 ns).
 * decomoe_selftest_wait launches one kernel that waits on a device barrier
 * nothing ever completes, with the given limit, so that the timeout path can
 * be tested without faulting or hanging the GPU.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_read_status(int32_t* status_dev, int32_t* code_host, decomoe_stream_t stream);
DECOMOE_API int decomoe_set_wait_limit_ns(int64_t limit_ns);
DECOMOE_API int decomoe_selftest_wait(int32_t* status_dev, int64_t limit_ns, decomoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Scratch lines in L2. With on != 0 (the default), decomoe_moe_layer and
 * decomoe_moe_layer_exit drop the L2 lines of their workspace's y_perm rows
 * once the combine has read them (discard.global.L2): the rows are not
 * written back to HBM, and the next layer's writes find clean lines to
 * evict. Those workspace rows are undefined after the call. on == 0 keeps
 * them (for inspection). Process-wide; applies to later calls.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_set_discard_scratch(int on);

/* ------------------------------------------------------------------------
 * Programmatic dependent launch. With on != 0 (the default) kernels of at
 * most one block per SM are launched so that their blocks are scheduled while
 * the previous kernel on the stream drains; each waits (griddepcontrol.wait)
 * before it reads what earlier kernels wrote, so results are the same bits
 * either way. on == 0 launches every kernel plainly. Process-wide; applies
 * to later launches and to graphs captured after the call.
 * ------------------------------------------------------------------------ */
DECOMOE_API int decomoe_set_pdl(int on);

#ifdef __cplusplus
}
#endif

#endif /* DECOMOE_H */
