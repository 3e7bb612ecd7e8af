// Internal launchers of the fingerprint kernels.  The C entry points of
// fp_ops.h and the runtime of fp.h both go through these; arguments are
// validated by the callers, so the launchers only launch.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/fp_ops.h"

namespace fpk {

// ---- weights: seeded fill and quantisers (fp_quant.cu)
cudaError_t launch_init_weights(uint16_t* w, long long n, unsigned long long seed, long long stream_id,
                                long long start, cudaStream_t s);
// perm: the act order of a GPTQ4 matrix (ignored for the other formats)
cudaError_t launch_quantize(int wquant, const uint16_t* w, int N, int K, void* codes, uint16_t* scales,
                            uint16_t* zeros, cudaStream_t s, const int32_t* perm = nullptr);
// xp[m][j] = x[m][perm[j]] (K % 8 == 0); inv[perm[j]] = j.  Entries of perm
// outside [0, K) set *err = 1 (err may be NULL).
cudaError_t launch_gather_cols(const uint16_t* x, int M, int K, const int32_t* perm, uint16_t* xp, int32_t* err,
                               cudaStream_t s);
cudaError_t launch_invert_perm(const int32_t* perm, int K, int32_t* inv, int32_t* err, cudaStream_t s);

// ---- small row kernels (fp_rows.cu)
cudaError_t launch_embed(const int32_t* tok, int M, const uint16_t* E, int V, int d, uint16_t* h,
                         int32_t* err, cudaStream_t s);
cudaError_t launch_rmsnorm(const uint16_t* x, int M, int d, int row_stride, int row_offset,
                           const uint16_t* g, float eps, uint16_t* y, cudaStream_t s);
// pos (optional): pos[row] += by once row's token is written.
cudaError_t launch_argmax(const float* logits, int M, int V, int32_t* out, cudaStream_t s, int32_t* pos = nullptr,
                          int by = 0);
cudaError_t launch_embed_rmsnorm(const int32_t* tok, int M, const uint16_t* E, int V, int d, uint16_t* h,
                                 const uint16_t* g, float eps, uint16_t* y, int32_t* err, cudaStream_t s);
cudaError_t launch_rope_kv(uint16_t* qkv, int B, int S, int row_stride, int n_heads, const fp_kv_view& kv,
                           const int32_t* pos, const float* rope_cs, int32_t* err, cudaStream_t s);

// ---- attention (fp_attention.cu)
size_t attention_decode_ws_bytes(int B, int n_heads, int head_dim, int max_len);
// Kernels one decode-attention launch runs: 1 (one split, normalised in place) or 2 (splits + combine).
int attention_decode_launches(int B, int n_kv_heads, int head_dim, int kvquant, int max_len);
// Context splits of one decode-attention launch (1: the partials workspace is not touched).
int attention_decode_splits(int B, int n_kv_heads, int head_dim, int kvquant, int max_len);
cudaError_t launch_attention_decode(const uint16_t* q, int q_stride, int B, int n_heads, const fp_kv_view& kv,
                                    const int32_t* len, int len_add, int max_len, uint16_t* out, void* ws,
                                    int32_t* err, cudaStream_t s, cudaError_t* second = nullptr);
// tcgen05 prefill attention (bf16 cache, head_dim 128, 16-token pages; fp_attn_tc.cu)
bool attention_prefill_tc_ok(int B, int S, int n_heads, const fp_kv_view& kv, const void* q, int q_stride);
cudaError_t launch_attention_prefill_tc(const uint16_t* q, int q_stride, int B, int S, int n_heads,
                                        const fp_kv_view& kv, uint16_t* out, int32_t* err, cudaStream_t s);
cudaError_t launch_attention_prefill(const uint16_t* q, int q_stride, int B, int S, int n_heads,
                                     const fp_kv_view& kv, uint16_t* out, int32_t* err, cudaStream_t s);

// ---- weight-only linear (fp_linear.cu)
// Split-K ticket counters at the head of a linear's workspace (zero at rest).
constexpr int kLinTicketSlots = 4096;
// Workspace of one launch with exactly these M, N, K (any epilogue); 0 if none.
size_t linear_ws_bytes(int wquant, int M, int N, int K);
// Largest workspace over every M in [1, max_m].
size_t linear_ws_bytes_upto(int wquant, int max_m, int N, int K);
cudaError_t launch_linear(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                          const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                          void* ws, size_t ws_bytes, cudaStream_t s, int32_t* err = nullptr);

// GPTQ4 linear (fp_linear.cu): decode gathers x into the act order, prefill
// expands the weights back into channel order.  inv may be NULL (computed
// into the workspace, which is then K * 4 bytes larger for M > 64).
size_t linear_gptq4_ws_bytes(int M, int N, int K, bool with_inv);
size_t linear_gptq4_ws_bytes_upto(int max_m, int N, int K, bool with_inv);
cudaError_t launch_linear_gptq4(int epi, const uint16_t* x, int M, int N, int K, const int32_t* perm,
                                const int32_t* inv, const void* codes, const uint16_t* scales,
                                const uint16_t* zeros, const uint16_t* residual, void* y, void* ws, size_t ws_bytes,
                                cudaStream_t s, int32_t* err);

// ---- int4 / int8 decode linear at 17-64 tokens on tcgen05 (fp_gemv_tc.cu)
bool q4tc_ok(int wquant, int epi, int M, int N, int K);
bool q4tc_preferred(int wquant, int M, int K);
size_t q4tc_ws_bytes(int epi, int M, int N, int K);
cudaError_t launch_q4tc(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                        const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y, void* ws,
                        size_t ws_bytes, int32_t* err, cudaStream_t s);

// ---- bf16 decode linear at 17-64 tokens on tcgen05, TMA-fed (fp_gemv_btc.cu)
bool btc_ok(int wquant, int epi, int M, int N, int K);
bool btc_preferred(int epi, int N, int K);  // enough work per SM for the TMA-fed kernel
size_t btc_ws_bytes(int epi, int M, int N, int K);
cudaError_t launch_btc(int epi, const uint16_t* x, int M, int N, int K, const void* w, const uint16_t* residual,
                       void* y, void* ws, size_t ws_bytes, int32_t* err, cudaStream_t s);

// ---- prefill GEMM on tcgen05 (fp_gemm_tc.cu)
bool gemm_tc_ok(int M, int N, int K);
size_t gemm_tc_ws_bytes(int wquant, int N, int K);
// inv: the inverse act order of a GPTQ4 matrix (its expansion returns to channel order)
cudaError_t launch_gemm_tc(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                           const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                           void* ws, size_t ws_bytes, int32_t* err, cudaStream_t s, const int32_t* inv = nullptr);

// ---- prefill GEMM with int8 / int4 weights dequantised in the kernel (fp_gemm_wq.cu)
bool gemm_wq_ok(int wquant, int epi, int M, int N, int K, const void* x, const void* codes);
cudaError_t launch_gemm_wq(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                           const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                           int32_t* err, cudaStream_t s);

}  // namespace fpk
