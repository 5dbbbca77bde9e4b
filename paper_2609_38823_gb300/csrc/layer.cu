// One RCEP MoE invocation chained on a stream (DecoMoE Algorithm 2, exited
// branch): router logits over the full pool, the activated-mass pass and
// prefix selection (Eqs. 10-12), prefix routing, dispatch, grouped SwiGLU
// experts and combine. Every intermediate lives in the caller's workspace.
#include <vector>

#include "decomoe_internal.cuh"

namespace decomoe {

enum {
  WS_LOGITS = 0,
  WS_TOPK_IDX,
  WS_TOPK_W,
  WS_MASS,
  WS_COUNTS,
  WS_OFFSETS,
  WS_PERM,
  WS_INV,
  WS_XPERM,
  WS_H,
  WS_YPERM,
  WS_ROUTE,
  WS_KDEV,
  WS_SCHED,
  WS_RSPLIT,
  WS_SYNC,
  WS_DSYNC,
  WS_STATUS_PAD,
  WS_COUNT
};

// a2-a5 over logits read through src (plain logits, or the k-split
// router's partial sums): mass pass, prefix (fixed, or Eq. 12 on the
// device), prefix routing and dispatch. With a fixed prefix and mass_out the
// activated mass is finished by the dispatch launch's extra blocks.
static int route_dispatch_src(const float* logits, const RouteSrc& src, int64_t T, int E, int K, int k, double p,
                              int32_t* topk_idx, float* topk_w, double* mass_out, int32_t* K_dev, const void* x,
                              int d, int dtype, int32_t* counts, int32_t* offsets, int32_t* perm_token,
                              int32_t* inv_slot, void* x_perm, void* ws, size_t ws_bytes, int32_t* status_dev,
                              cudaStream_t s, int32_t* zero_ints = nullptr, int n_zero = 0) {
  DM_ARG_CHECK(T >= 0, "route_dispatch: T < 0");
  DM_ARG_CHECK(E >= 1 && E <= DECOMOE_MAX_E && k >= 1 && k <= DECOMOE_MAX_TOPK && k <= E,
               "route_dispatch: need 1 <= k <= E <= %d, k <= %d", DECOMOE_MAX_E, DECOMOE_MAX_TOPK);
  const bool device_k = (K == -1);
  DM_ARG_CHECK(device_k || (K >= k && K <= E), "route_dispatch: need k <= K <= E or K = -1 (k=%d K=%d E=%d)", k,
               K, E);
  if (device_k) {
    DM_ARG_CHECK(p > 0.0 && p <= 1.0, "route_dispatch: a device-selected prefix needs 0 < p <= 1");
    DM_ARG_CHECK(mass_out && K_dev, "route_dispatch: a device-selected prefix needs mass_out and K_dev");
  }
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "route_dispatch: bad dtype");
  DM_ARG_CHECK(counts && offsets, "route_dispatch: counts/offsets null");
  const int Kd = device_k ? E : K;
  decomoe_stream_t stream = reinterpret_cast<decomoe_stream_t>(s);
  if (T == 0) {
    DM_CUDA_CHECK(cudaMemsetAsync(counts, 0, sizeof(int32_t) * Kd, s));
    DM_CUDA_CHECK(cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (Kd + 1), s));
    if (mass_out) DM_CUDA_CHECK(cudaMemsetAsync(mass_out, 0, sizeof(double) * E, s));
    if (device_k) return decomoe_select_prefix_device(mass_out, E, k, p, K_dev, stream);  // zero mass: K = k
    return DECOMOE_OK;
  }
  DM_ARG_CHECK(logits && topk_idx && topk_w && perm_token && inv_slot, "route_dispatch: null pointer");
  DM_ARG_CHECK(T * static_cast<int64_t>(k) < 0x7fffffffLL, "route_dispatch: T*k too large");
  const size_t row_bytes = static_cast<size_t>(d) * dtype_bytes(dtype);
  if (x_perm != nullptr) {
    DM_ARG_CHECK(x != nullptr && d > 0, "route_dispatch: x null or d <= 0");
    DM_ARG_CHECK(row_bytes % 16 == 0 && aligned16(x) && aligned16(x_perm),
                 "route_dispatch: rows must be 16-byte multiples and 16-byte aligned");
  }
  const size_t rbytes = align_up(decomoe_route_workspace_bytes(T, E), 256);
  const size_t dbytes = decomoe_dispatch_workspace_bytes(T, k, E);
  if (ws == nullptr || ws_bytes < rbytes + dbytes) {
    set_error("route_dispatch: workspace needs %zu bytes", rbytes + dbytes);
    return DECOMOE_ERR_WORKSPACE;
  }
  void* route_ws = ws;
  void* disp_ws = static_cast<uint8_t*>(ws) + rbytes;
  int mass_blocks = 0;
  // decode sizes (one routing block): that block also counts, ranks and, for
  // up to 64 KiB of rows, gathers its picks; larger rows are copied by the
  // gather launch
  const bool one_block = T <= ROUTE_TOKENS_PER_BLOCK;
  RouteDispatch rd;
  if (one_block) {
    rd.counts = counts;
    rd.offsets = offsets;
    rd.perm_token = perm_token;
    rd.inv_slot = inv_slot;
    rd.status = status_dev;
    rd.x = x;
    rd.row_vec = static_cast<int>(row_bytes / 16);
    rd.x_perm = (x_perm != nullptr && static_cast<size_t>(T) * k * row_bytes <= 64 * 1024) ? x_perm : nullptr;
    rd.Kd = Kd;
  }
  if (device_k) {
    // mass pass, Eq. 12 on the device, routing over [0, *K_dev) (from the
    // summed logits when the first pass read the router's partials)
    DM_RET(route_prefix_src(logits, src, T, E, E, E, k, nullptr, nullptr, mass_out, route_ws, rbytes, false, nullptr,
                            s, nullptr, nullptr, zero_ints, n_zero));
    DM_RET(decomoe_select_prefix_device(mass_out, E, k, p, K_dev, stream));
    DM_RET(route_prefix_src(src.logits_out != nullptr ? src.logits_out : logits, RouteSrc{}, T, E, E, E, k, topk_idx,
                            topk_w, nullptr, nullptr, 0, false, nullptr, s, K_dev, one_block ? &rd : nullptr));
  } else {
    // one launch: prefix routing and, with mass_out, the full-pool partial
    // masses (finished by the dispatch launch)
    DM_RET(route_prefix_src(logits, src, T, E, E, K, k, topk_idx, topk_w, mass_out, route_ws, rbytes, true,
                            &mass_blocks, s, nullptr, one_block ? &rd : nullptr, zero_ints, n_zero));
  }
  if (one_block) {
    // one routing block: the mass was written in place and the picks are dispatched
    if (x_perm != nullptr && rd.x_perm == nullptr)
      DM_RET(launch_gather_rows(x, perm_token, offsets, Kd, row_bytes, T * k, x_perm, s));
    return DECOMOE_OK;
  }
  return dispatch_with_mass(topk_idx, T, k, Kd, x, d, dtype, counts, offsets, perm_token, inv_slot, x_perm, disp_ws,
                            dbytes, status_dev, mass_blocks > 0 ? static_cast<const double*>(route_ws) : nullptr,
                            mass_blocks, E, mass_out, s);
}

// a1-a5: router logits (as partial sums read by the routing kernel when the
// router splits its k loop, else written out first), then route_dispatch_src.
// scratch: the split router's partials (decomoe_router_logits_ws_bytes).
static int router_route_dispatch_impl(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E,
                                      int dtype, int K, int k, double p, float* logits, int32_t* topk_idx,
                                      float* topk_w, double* mass_out, int32_t* K_dev, int32_t* counts,
                                      int32_t* offsets, int32_t* perm_token, int32_t* inv_slot, void* x_perm,
                                      float* scratch, void* rd_ws, size_t rd_bytes, int32_t* status_dev,
                                      cudaStream_t s, int32_t* zero_ints = nullptr, int n_zero = 0) {
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "router_route_dispatch: bad dtype");
  RouteSrc src;
  const float* lg = logits;
  if (T > 0) {
    DM_ARG_CHECK(x && w_r && logits, "router_route_dispatch: null pointer");
    int ks = 1;
    const size_t split_bytes = dtype == DECOMOE_BF16 ? decomoe_router_logits_ws_bytes(T, d, E) : 0;
    if (split_bytes > 0 && aligned16(x) && aligned16(w_r) && aligned16(scratch) && aligned16(logits) &&
        (bias == nullptr || aligned16(bias)))
      DM_RET(launch_router_parts(x, w_r, T, d, E, scratch, status_dev, s, &ks));
    if (ks > 1) {
      src.nparts = ks;
      src.part_stride = T * E;
      src.bias = bias;
      src.logits_out = logits;
      lg = scratch;
    } else {
      // unsplit router, or operands the slice-reading routing kernel cannot
      // take: the logits first, exactly as decomoe_router_logits_ws forms them
      DM_RET(decomoe_router_logits_ws(x, w_r, bias, T, d, E, dtype, logits, scratch, split_bytes, status_dev,
                                      reinterpret_cast<decomoe_stream_t>(s)));
    }
  }
  return route_dispatch_src(lg, src, T, E, K, k, p, topk_idx, topk_w, mass_out, K_dev, x, d, dtype, counts, offsets,
                            perm_token, inv_slot, x_perm, rd_ws, rd_bytes, status_dev, s, zero_ints, n_zero);
}

struct LayerLayout {
  size_t off[WS_COUNT];
  size_t total;
};

static LayerLayout layer_layout(int64_t T, int d, int E, int k, int m, int dtype) {
  LayerLayout L;
  const size_t eb = dtype_bytes(dtype);
  const size_t R = static_cast<size_t>(T) * k;
  size_t sz[WS_COUNT];
  sz[WS_LOGITS] = static_cast<size_t>(T) * E * 4;
  sz[WS_TOPK_IDX] = R * 4;
  sz[WS_TOPK_W] = R * 4;
  sz[WS_MASS] = static_cast<size_t>(E) * 8;
  sz[WS_COUNTS] = static_cast<size_t>(E) * 4;
  sz[WS_OFFSETS] = static_cast<size_t>(E + 1) * 4;
  sz[WS_PERM] = R * 4;
  sz[WS_INV] = R * 4;
  sz[WS_XPERM] = R * d * eb;
  sz[WS_H] = R * m * eb;
  sz[WS_YPERM] = R * d * eb;
  sz[WS_ROUTE] = decomoe_route_dispatch_workspace_bytes(T, k, E);
  sz[WS_KDEV] = 16;
  sz[WS_SCHED] = 16;
  sz[WS_RSPLIT] = decomoe_router_logits_ws_bytes(T, d, E);
  sz[WS_SYNC] = expert_ffn_sync_ints(static_cast<int64_t>(T) * k, E) * 4;  // counters of the fused expert launch
  sz[WS_DSYNC] = decode_layer_sync_ints(T, d, E) * 4;  // counters of the one-launch decode layer
  sz[WS_STATUS_PAD] = 256;
  size_t o = 0;
  for (int i = 0; i < WS_COUNT; ++i) {
    L.off[i] = o;
    o = align_up(o + sz[i], 256);
  }
  L.total = o;
  return L;
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

size_t decomoe_moe_layer_workspace_bytes(int64_t T, int d, int E, int k, int m, int dtype) {
  if (T < 0 || d <= 0 || E <= 0 || k <= 0 || m <= 0) return 0;
  return layer_layout(T, d, E, k, m, dtype).total;
}

int decomoe_moe_layer_workspace_layout(int64_t T, int d, int E, int k, int m, int dtype, size_t* offs_host) {
  clear_error();
  DM_ARG_CHECK(offs_host != nullptr, "moe_layer_workspace_layout: null pointer");
  DM_ARG_CHECK(T >= 0 && d > 0 && E > 0 && k > 0 && m > 0, "moe_layer_workspace_layout: bad sizes");
  const LayerLayout L = layer_layout(T, d, E, k, m, dtype);
  for (int i = 0; i <= WS_YPERM; ++i) offs_host[i] = L.off[i];
  offs_host[11] = L.off[WS_KDEV];
  return DECOMOE_OK;
}

size_t decomoe_route_dispatch_workspace_bytes(int64_t T, int k, int E) {
  if (T < 0 || k <= 0 || E <= 0) return 0;
  return align_up(decomoe_route_workspace_bytes(T, E), 256) + decomoe_dispatch_workspace_bytes(T, k, E);
}

int decomoe_route_dispatch(const float* logits, int64_t T, int E, int K, int k, double p, int32_t* topk_idx,
                           float* topk_w, double* mass_out, int32_t* K_dev, const void* x, int d, int dtype,
                           int32_t* counts, int32_t* offsets, int32_t* perm_token, int32_t* inv_slot, void* x_perm,
                           void* ws, size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream) {
  clear_error();
  return route_dispatch_src(logits, RouteSrc{}, T, E, K, k, p, topk_idx, topk_w, mass_out, K_dev, x, d, dtype,
                            counts, offsets, perm_token, inv_slot, x_perm, ws, ws_bytes, status_dev,
                            reinterpret_cast<cudaStream_t>(stream));
}

size_t decomoe_router_route_dispatch_workspace_bytes(int64_t T, int d, int E, int k) {
  if (T < 0 || d <= 0 || E <= 0 || k <= 0) return 0;
  return align_up(decomoe_router_logits_ws_bytes(T, d, E), 256) + decomoe_route_dispatch_workspace_bytes(T, k, E);
}

int decomoe_router_route_dispatch(const void* x, const void* w_r, const float* bias, int64_t T, int d, int E,
                                  int dtype, int K, int k, double p, float* logits, int32_t* topk_idx, float* topk_w,
                                  double* mass_out, int32_t* K_dev, int32_t* counts, int32_t* offsets,
                                  int32_t* perm_token, int32_t* inv_slot, void* x_perm, void* ws, size_t ws_bytes,
                                  int32_t* status_dev, decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(T >= 0 && d > 0, "router_route_dispatch: bad sizes");
  const size_t rs = align_up(decomoe_router_logits_ws_bytes(T, d, E), 256);
  const size_t need = decomoe_router_route_dispatch_workspace_bytes(T, d, E, k);
  if (T > 0 && (ws == nullptr || ws_bytes < need)) {
    set_error("router_route_dispatch: workspace needs %zu bytes", need);
    return DECOMOE_ERR_WORKSPACE;
  }
  return router_route_dispatch_impl(x, w_r, bias, T, d, E, dtype, K, k, p, logits, topk_idx, topk_w, mass_out, K_dev,
                                    counts, offsets, perm_token, inv_slot, x_perm,
                                    T > 0 ? static_cast<float*>(ws) : nullptr,
                                    T > 0 ? static_cast<uint8_t*>(ws) + rs : nullptr, T > 0 ? ws_bytes - rs : 0,
                                    status_dev, reinterpret_cast<cudaStream_t>(stream));
}

int decomoe_moe_layer(const void* x, const void* w_r, const float* bias, const void* w_gate_up,
                      const void* w_down, int64_t T, int d, int E, int k, int m, int dtype, int K_fixed,
                      double p, const void* residual, void* out, int* K_used_host, int* K_sel_host, void* ws,
                      size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream) {
  clear_error();
  return moe_layer_impl(x, w_r, bias, w_gate_up, w_down, T, d, E, k, m, dtype, K_fixed, p, residual, out, nullptr,
                        0, 0, K_used_host, K_sel_host, ws, ws_bytes, status_dev, stream);
}

int decomoe_moe_layer_exit(const void* x, const void* w_r, const float* bias, const void* w_gate_up,
                           const void* w_down, int64_t T, int d, int E, int k, int m, int dtype, int K_fixed,
                           double p, const void* residual, void* out, void* text_out, int64_t v0, int64_t nv,
                           int* K_used_host, int* K_sel_host, void* ws, size_t ws_bytes, int32_t* status_dev,
                           decomoe_stream_t stream) {
  clear_error();
  DM_ARG_CHECK(v0 >= 0 && nv >= 0 && v0 + nv <= T, "moe_layer_exit: visual block [%lld, %lld) outside [0, %lld)",
               (long long)v0, (long long)(v0 + nv), (long long)T);
  DM_ARG_CHECK(text_out != nullptr || T - nv == 0, "moe_layer_exit: text_out is null");
  return moe_layer_impl(x, w_r, bias, w_gate_up, w_down, T, d, E, k, m, dtype, K_fixed, p, residual, out,
                        T - nv > 0 ? text_out : nullptr, v0, nv, K_used_host, K_sel_host, ws, ws_bytes, status_dev,
                        stream);
}

}  // extern "C"

namespace decomoe {

int moe_layer_impl(const void* x, const void* w_r, const float* bias, const void* w_gate_up, const void* w_down,
                   int64_t T, int d, int E, int k, int m, int dtype, int K_fixed, double p, const void* residual,
                   void* out, void* text_out, int64_t v0, int64_t nv, int* K_used_host, int* K_sel_host, void* ws,
                   size_t ws_bytes, int32_t* status_dev, decomoe_stream_t stream) {
  DM_ARG_CHECK(T >= 0 && d > 0 && m > 0, "moe_layer: bad sizes");
  DM_ARG_CHECK(E >= 1 && E <= DECOMOE_MAX_E && k >= 1 && k <= DECOMOE_MAX_TOPK && k <= E,
               "moe_layer: need 1 <= k <= E <= %d, k <= %d", DECOMOE_MAX_E, DECOMOE_MAX_TOPK);
  DM_ARG_CHECK(K_fixed == 0 || K_fixed == -1 || (K_fixed >= k && K_fixed <= E),
               "moe_layer: K_fixed=%d outside [k, E] (0: host-selected, -1: device-selected)", K_fixed);
  DM_ARG_CHECK(K_fixed > 0 || (p > 0.0 && p <= 1.0), "moe_layer: mass mode needs 0 < p <= 1");
  DM_ARG_CHECK(p >= 0.0 && p <= 1.0, "moe_layer: p outside [0, 1]");
  DM_ARG_CHECK(dtype == DECOMOE_BF16 || dtype == DECOMOE_F32, "moe_layer: bad dtype");
  // the expert call's shape rules, checked before the first launch
  DM_ARG_CHECK(m % DECOMOE_GU_BLOCK == 0, "moe_layer: m must be a multiple of %d", DECOMOE_GU_BLOCK);
  DM_ARG_CHECK(dtype != DECOMOE_BF16 || (m % 128 == 0 && d % 256 == 0),
               "moe_layer: bf16 needs m %% 128 == 0 and d %% 256 == 0 (m=%d, d=%d)", m, d);
  if (T == 0) {
    if (K_used_host) *K_used_host = K_fixed > 0 ? K_fixed : k;
    if (K_sel_host) *K_sel_host = k;
    return DECOMOE_OK;
  }
  DM_ARG_CHECK(x && w_r && w_gate_up && w_down && out, "moe_layer: null pointer");
  DM_ARG_CHECK(out != x, "moe_layer: out aliases x");
  const LayerLayout L = layer_layout(T, d, E, k, m, dtype);
  if (ws == nullptr || ws_bytes < L.total) {
    set_error("moe_layer: workspace needs %zu bytes", L.total);
    return DECOMOE_ERR_WORKSPACE;
  }
  DM_ARG_CHECK(aligned16(ws), "moe_layer: workspace must be 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint8_t* base = static_cast<uint8_t*>(ws);
  float* logits = reinterpret_cast<float*>(base + L.off[WS_LOGITS]);
  int32_t* topk_idx = reinterpret_cast<int32_t*>(base + L.off[WS_TOPK_IDX]);
  float* topk_w = reinterpret_cast<float*>(base + L.off[WS_TOPK_W]);
  double* mass = reinterpret_cast<double*>(base + L.off[WS_MASS]);
  int32_t* counts = reinterpret_cast<int32_t*>(base + L.off[WS_COUNTS]);
  int32_t* offsets = reinterpret_cast<int32_t*>(base + L.off[WS_OFFSETS]);
  int32_t* perm = reinterpret_cast<int32_t*>(base + L.off[WS_PERM]);
  int32_t* inv = reinterpret_cast<int32_t*>(base + L.off[WS_INV]);
  void* x_perm = base + L.off[WS_XPERM];
  void* h = base + L.off[WS_H];
  void* y_perm = base + L.off[WS_YPERM];
  void* route_ws = base + L.off[WS_ROUTE];  // routing and dispatch scratch

  int K = K_fixed;
  int32_t* K_dev = reinterpret_cast<int32_t*>(base + L.off[WS_KDEV]);
  float* rsplit = reinterpret_cast<float*>(base + L.off[WS_RSPLIT]);
  // counters of the fused expert launch (per expert or per M-tile), cleared
  // by the first routing launch of this call
  int32_t* sync = reinterpret_cast<int32_t*>(base + L.off[WS_SYNC]);
  const int n_sync = static_cast<int>(expert_ffn_sync_ints(T * k, E));
  // Decode sizes: the whole layer as one launch (router, routing, dispatch,
  // experts and combine; its counters in their own workspace slot).
  if (decode_layer_supported(T, d, E, k, m, dtype, K_fixed)) {
    if (K_used_host) *K_used_host = K_fixed;
    if (K_sel_host && K_fixed == -1) *K_sel_host = -1;
    return launch_decode_layer(x, w_r, bias, w_gate_up, w_down, T, d, E, k, m, K_fixed, p, residual, out, text_out,
                               v0, nv, logits,
                               topk_idx, topk_w, mass, counts, offsets, perm, inv, x_perm, h, y_perm, K_dev,
                               reinterpret_cast<int32_t*>(base + L.off[WS_DSYNC]), status_dev, s);
  }
  // Where the experts take the one-launch tokens-as-M form on at least
  // gather_min_rows routed rows, that launch copies the
  // dispatched rows itself (per M-tile, while its accumulators fill) and the
  // dispatch skips its gather launch (measured: T=2048 K=64 0.2258 -> 0.2244
  // ms, end to end 8.80 -> 9.00 M tokens/s; at 1024 rows 3.4 us slower, the
  // shares being a few rows each).
  constexpr int64_t gather_min_rows = 8192;
  auto ffn_gathers = [&](int K_groups) {
    return T * k >= gather_min_rows && expert_ffn_fused_kind(T * k, K_groups, m, dtype) == FFN_FUSED_TC;
  };
  bool gathers = false;
  if (K_fixed != 0) {
    // a1-a5: router logits over all E reordered experts, full-pool mass
    // (Eq. 11), prefix (fixed, or Eq. 12 on the device), prefix routing and
    // dispatch; with a device-selected prefix, dispatch and the experts run
    // over all E groups (those at or beyond *K_dev are empty)
    gathers = ffn_gathers(K_fixed == -1 ? E : K_fixed);
    DM_RET(router_route_dispatch_impl(x, w_r, bias, T, d, E, dtype, K_fixed, k, p, logits, topk_idx, topk_w,
                                      (K_fixed == -1 || p > 0.0) ? mass : nullptr, K_dev, counts, offsets, perm, inv,
                                      gathers ? nullptr : x_perm, rsplit, route_ws, L.off[WS_KDEV] - L.off[WS_ROUTE],
                                      status_dev, s, sync, n_sync));
    if (K_fixed == -1) {
      K = E;
      if (K_sel_host) *K_sel_host = -1;
      if (K_used_host) *K_used_host = -1;
    }
  } else {
    // host-selected prefix: router logits, mass pass, one device-to-host
    // read, Eq. 12 in C
    DM_RET(decomoe_router_logits_ws(x, w_r, bias, T, d, E, dtype, logits, rsplit,
                                    decomoe_router_logits_ws_bytes(T, d, E), status_dev, stream));
    DM_RET(route_prefix_src(logits, RouteSrc{}, T, E, E, E, k, nullptr, nullptr, mass, route_ws,
                            decomoe_route_workspace_bytes(T, E), false, nullptr, s, nullptr, nullptr, sync, n_sync));
    static thread_local std::vector<double> h_mass;
    h_mass.resize(E);
    DM_CUDA_CHECK(cudaMemcpyAsync(h_mass.data(), mass, sizeof(double) * E, cudaMemcpyDeviceToHost, s));
    DM_CUDA_CHECK(cudaStreamSynchronize(s));
    int Ksel = k;
    DM_RET(decomoe_select_prefix(h_mass.data(), E, k, p, &Ksel));
    K = Ksel;
    if (K_sel_host) *K_sel_host = Ksel;
    gathers = ffn_gathers(K);
    DM_RET(decomoe_route_dispatch(logits, T, E, K, k, 0.0, topk_idx, topk_w, nullptr, nullptr, x, d, dtype, counts,
                                  offsets, perm, inv, gathers ? nullptr : x_perm, route_ws,
                                  L.off[WS_KDEV] - L.off[WS_ROUTE], status_dev, stream));
  }
  if (K_used_host && K_fixed != -1) *K_used_host = K;
  // a6: grouped SwiGLU experts over [0, K): at decode sizes gate/up and down
  // in one launch, else the two GEMMs (static tile order: as fast as the
  // dynamic queue here, and no counter reset between the launches, which
  // keeps them chained programmatically)
  bool fused = false;
  DM_RET(launch_expert_ffn_fused(x_perm, offsets, T * k, K, d, m, dtype, w_gate_up, w_down, h, y_perm, sync,
                                 status_dev, s, &fused, gathers ? x : nullptr, gathers ? perm : nullptr));
  if (!fused)
    DM_RET(decomoe_expert_swiglu(x_perm, offsets, T * k, K, d, m, dtype, w_gate_up, w_down, h, y_perm, status_dev,
                                 nullptr, stream));
  // a7: combine (+ residual); with text_out also a8 on the layer output
  // y_perm is the call's own scratch: its lines leave L2 without a write-back
  return combine_impl(y_perm, inv, topk_w, T, k, d, dtype, residual, out, text_out, v0, nv, stream,
                      discard_scratch());
}

}  // namespace decomoe
