// Latency and memory estimators of the profiling method (Sec. 5.2-5.3):
// Eq. 1 fitted per fingerprint from two output lengths, Eqs. 2-3 from two
// fingerprint depths, and the linear memory extrapolation.  Host code; each
// 2x2 system is solved by Cramer's rule (determinant != 0 is the only
// condition, checked exactly on the integer coefficients).
#include "fp.h"
#include "fp_estimate.h"

extern "C" int fp_solve_eq1(int len_a, double lat_a, int len_b, double lat_b, fp_eq1_fit* out) {
  if (!out || len_a == len_b) return FP_ERR_INVALID_ARG;
  // [1 len_a; 1 len_b] [ttft; tpot] = [lat_a; lat_b]
  const double det = (double)len_b - (double)len_a;
  const double tpot = (lat_b - lat_a) / det;
  out->tpot = tpot;
  out->ttft = lat_a - len_a * tpot;
  return FP_OK;
}

extern "C" int fp_solve_eq23(int layers_a, const fp_eq1_fit* a, int layers_b, const fp_eq1_fit* b, fp_l2_terms* out) {
  if (!a || !b || !out || layers_a == layers_b) return FP_ERR_INVALID_ARG;
  const double det = (double)layers_b - (double)layers_a;
  // [layers_a 1; layers_b 1] [x_layer; x_other] = [x_a; x_b], for x = TTFT and x = TPOT
  const double ttft_layer = (b->ttft - a->ttft) / det;
  const double tpot_layer = (b->tpot - a->tpot) / det;
  out->ttft_layer = ttft_layer;
  out->ttft_other = a->ttft - layers_a * ttft_layer;
  out->tpot_layer = tpot_layer;
  out->tpot_other = a->tpot - layers_a * tpot_layer;
  return FP_OK;
}

extern "C" int fp_predict_latency(const fp_l2_terms* t, int num_layers, int output_length, double* latency) {
  if (!t || !latency) return FP_ERR_INVALID_ARG;
  const double ttft = num_layers * t->ttft_layer + t->ttft_other;
  const double tpot = num_layers * t->tpot_layer + t->tpot_other;
  *latency = ttft + output_length * tpot;
  return FP_OK;
}

extern "C" int fp_extrapolate_memory(int layers_a, double mem_a, int layers_b, double mem_b, int num_layers,
                                     double* mem) {
  if (!mem || layers_a == layers_b) return FP_ERR_INVALID_ARG;
  const double slope = (mem_b - mem_a) / ((double)layers_b - (double)layers_a);
  *mem = mem_a + slope * (num_layers - layers_a);
  return FP_OK;
}
