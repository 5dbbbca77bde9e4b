/* Host-side prefix selection of RCEP (DecoMoE Section 3.3, Eq. 12), plain C.
 *
 * K_hat = min{K in 1..E : sum_{e<K} mass[e] / sum_e mass[e] >= p},
 * K     = max(k, K_hat).
 * The sums run sequentially over e = 0..E-1 in double precision and the total
 * is the last partial sum, so the result depends only on the mass values.
 * The paper leaves three cases open; the readings taken: p == 1 keeps the
 * whole pool (its sweep reports a prefix of 128.0 of 128 at p = 1.0), a ratio
 * that never reaches p through rounding also keeps the whole pool, and an
 * invocation without routed mass (total 0) keeps k experts.
 */
#include <math.h>
#include <stddef.h>

#include "../../include/decomoe.h"

void decomoe_internal_set_error(const char* msg);

int decomoe_select_prefix(const double* mass_host, int E, int k, double p, int* K_out_host) {
  if (mass_host == NULL || K_out_host == NULL) {
    decomoe_internal_set_error("select_prefix: null pointer");
    return DECOMOE_ERR_INVALID_ARG;
  }
  if (E < 1 || k < 1 || k > E) {
    decomoe_internal_set_error("select_prefix: need 1 <= k <= E");
    return DECOMOE_ERR_INVALID_ARG;
  }
  if (!(p > 0.0 && p <= 1.0)) {
    decomoe_internal_set_error("select_prefix: p must lie in (0, 1]");
    return DECOMOE_ERR_INVALID_ARG;
  }
  double tot = 0.0;
  for (int e = 0; e < E; ++e) {
    if (!(mass_host[e] >= 0.0) || isinf(mass_host[e])) {
      decomoe_internal_set_error("select_prefix: mass must be finite and non-negative");
      return DECOMOE_ERR_INVALID_ARG;
    }
    tot = tot + mass_host[e];
  }
  if (!(tot > 0.0)) {
    *K_out_host = k;
    return DECOMOE_OK;
  }
  int K_hat = E;
  if (p < 1.0) {
    double acc = 0.0;
    for (int K = 1; K <= E; ++K) {
      acc = acc + mass_host[K - 1];
      if (acc / tot >= p) {
        K_hat = K;
        break;
      }
    }
  }
  *K_out_host = K_hat > k ? K_hat : k;
  return DECOMOE_OK;
}
