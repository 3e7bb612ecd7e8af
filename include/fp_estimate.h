/* Latency and memory estimators of the fingerprint profiling method
 * (arXiv 2501.13111, Sec. 5.2-5.3), on host doubles.  No GPU is involved:
 * the inputs are measurements, e.g. fp_profile_result.request_ms and
 * .peak_hbm_bytes of fingerprints with 1 and 2 hidden layers.
 *
 * Eq. 1  latency = TTFT + output_length * TPOT
 * Eq. 2  TTFT    = num_layers * TTFT_layer + TTFT_other
 * Eq. 3  TPOT    = num_layers * TPOT_layer + TPOT_other
 *
 * Every entry point returns 0 (FP_OK) or FP_ERR_INVALID_ARG (-1) for a
 * NULL pointer or a singular system (equal output lengths, equal layer
 * counts); outputs are written only on success.  Times are in whatever unit
 * the inputs use (ms for fp_profile). */
#ifndef FP_ESTIMATE_H
#define FP_ESTIMATE_H

#ifdef __cplusplus
extern "C" {
#endif

/* Eq. 1 fitted to one fingerprint: two requests of output lengths len_a and
 * len_b with latencies lat_a and lat_b (the 2x2 system of Sec. 5.3, L1). */
typedef struct fp_eq1_fit {
  double ttft, tpot;
} fp_eq1_fit;
int fp_solve_eq1(int len_a, double lat_a, int len_b, double lat_b, fp_eq1_fit* out);

/* Eqs. 2-3 from two fingerprints with layers_a != layers_b hidden layers
 * (Sec. 5.3, L2).  The 4x4 system of the paper decouples into one 2x2
 * system for TTFT and one for TPOT. */
typedef struct fp_l2_terms {
  double ttft_layer, ttft_other, tpot_layer, tpot_other;
} fp_l2_terms;
int fp_solve_eq23(int layers_a, const fp_eq1_fit* a, int layers_b, const fp_eq1_fit* b, fp_l2_terms* out);

/* Eq. 1 with Eqs. 2-3 substituted: the latency of a request of
 * output_length tokens on the model with num_layers hidden layers. */
int fp_predict_latency(const fp_l2_terms* t, int num_layers, int output_length, double* latency);

/* Memory (Sec. 5.2, TP = PP = 1): the footprint is linear in the number of
 * hidden layers, so two fingerprints give the footprint at num_layers. */
int fp_extrapolate_memory(int layers_a, double mem_a, int layers_b, double mem_b, int num_layers, double* mem);

#ifdef __cplusplus
}
#endif
#endif
