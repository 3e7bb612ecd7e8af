// C entry points of fp_ops.h: host-side argument checks, then one launcher
// of kernels.cuh.  Nothing here allocates.
#include <math.h>
#include <stdlib.h>

#include <vector>

#include "common.cuh"
#include "kernels.cuh"

using namespace fpk;

static int cuda_status(cudaError_t e) { return e == cudaSuccess ? FP_OK : FP_ERR_CUDA; }

static bool wquant_ok(int wq) { return wq == FP_W_BF16 || wq == FP_W_INT8 || wq == FP_W_INT4_G128; }

// K granularity of the weight formats: one 16-byte chunk of codes.
static int k_align(int wq) { return wq == FP_W_BF16 ? 8 : wq == FP_W_INT8 ? 16 : 128; }

int fpk_check_kv(const fp_kv_view* kv) {
  if (!kv || !kv->k_pool || !kv->v_pool || !kv->page_table) return FP_ERR_INVALID_ARG;
  if (kv->kvquant != FP_KV_BF16 && kv->kvquant != FP_KV_INT8) return FP_ERR_INVALID_ARG;
  if (kv->kvquant == FP_KV_INT8 && (!kv->k_scale || !kv->v_scale)) return FP_ERR_INVALID_ARG;
  if (kv->n_kv_heads <= 0 || kv->pages_per_seq <= 0 || kv->n_pages <= 0) return FP_ERR_INVALID_ARG;
  if (kv->head_dim != 64 && kv->head_dim != 128) return FP_ERR_UNSUPPORTED;
  if (kv->page_size != 16) return FP_ERR_UNSUPPORTED;
  return FP_OK;
}

extern "C" {

int fp_op_quantize(int wquant, const uint16_t* w, int N, int K, void* codes, uint16_t* scales, uint16_t* zeros,
                   void* stream) {
  if (!wquant_ok(wquant) || N < 0 || K <= 0 || !w || !codes) return FP_ERR_INVALID_ARG;
  if (wquant != FP_W_BF16 && !scales) return FP_ERR_INVALID_ARG;
  if (wquant == FP_W_INT4_G128 && !zeros) return FP_ERR_INVALID_ARG;
  if (wquant == FP_W_INT4_G128 && K % 128 != 0) return FP_ERR_UNSUPPORTED;
  return cuda_status(launch_quantize(wquant, w, N, K, codes, scales, zeros, (cudaStream_t)stream));
}

int fp_op_quantize_gptq4(const uint16_t* w, int N, int K, const int32_t* perm, void* codes, uint16_t* scales,
                         uint16_t* zeros, void* stream) {
  if (N < 0 || K <= 0 || !w || !perm || !codes || !scales || !zeros) return FP_ERR_INVALID_ARG;
  if (K % 128 != 0) return FP_ERR_UNSUPPORTED;
  return cuda_status(launch_quantize(FP_W_GPTQ4, w, N, K, codes, scales, zeros, (cudaStream_t)stream, perm));
}

size_t fp_op_linear_gptq4_workspace_bytes(int M, int N, int K) {
  if (M <= 0 || N <= 0 || K <= 0 || K % 128 != 0) return 0;
  return linear_gptq4_ws_bytes(M, N, K, true);
}

int fp_op_linear_gptq4(int epilogue, const uint16_t* x, int M, int N, int K, const int32_t* perm, const void* codes,
                       const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                       void* workspace, size_t workspace_bytes, int32_t* err, void* stream) {
  if (M < 0 || N <= 0 || K <= 0 || !x || !perm || !codes || !scales || !zeros || !y) return FP_ERR_INVALID_ARG;
  if (epilogue < FP_EPI_STORE || epilogue > FP_EPI_F32) return FP_ERR_INVALID_ARG;
  if (epilogue == FP_EPI_RESID && !residual) return FP_ERR_INVALID_ARG;
  if (epilogue == FP_EPI_SWIGLU && N % 2 != 0) return FP_ERR_INVALID_ARG;
  if (K % 128 != 0) return FP_ERR_UNSUPPORTED;
  if (M == 0) return FP_OK;
  if (!workspace || workspace_bytes < linear_gptq4_ws_bytes(M, N, K, true) || ((uintptr_t)workspace & 255))
    return FP_ERR_INVALID_ARG;
  return cuda_status(launch_linear_gptq4(epilogue, x, M, N, K, perm, nullptr, codes, scales, zeros, residual, y,
                                         workspace, workspace_bytes, (cudaStream_t)stream, err));
}

int fp_op_init_weights(uint16_t* w, long long n, unsigned long long seed, long long stream_id, long long start,
                       void* stream) {
  if (!w || n < 0 || start < 0) return FP_ERR_INVALID_ARG;
  return cuda_status(launch_init_weights(w, n, seed, stream_id, start, (cudaStream_t)stream));
}

size_t fp_op_linear_workspace_bytes(int wquant, int M, int N, int K) {
  if (!wquant_ok(wquant) || M <= 0 || N <= 0 || K <= 0) return 0;
  return linear_ws_bytes(wquant, M, N, K);
}

int fp_op_linear(int wquant, int epilogue, const uint16_t* x, int M, int N, int K, const void* codes,
                 const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y, void* workspace,
                 size_t workspace_bytes, void* stream) {
  if (!wquant_ok(wquant) || M < 0 || N <= 0 || K <= 0 || !x || !codes || !y) return FP_ERR_INVALID_ARG;
  if (epilogue < FP_EPI_STORE || epilogue > FP_EPI_F32) return FP_ERR_INVALID_ARG;
  if (wquant != FP_W_BF16 && !scales) return FP_ERR_INVALID_ARG;
  if (wquant == FP_W_INT4_G128 && !zeros) return FP_ERR_INVALID_ARG;
  if (epilogue == FP_EPI_RESID && !residual) return FP_ERR_INVALID_ARG;
  if (epilogue == FP_EPI_SWIGLU && N % 2 != 0) return FP_ERR_INVALID_ARG;
  if (K % k_align(wquant) != 0) return FP_ERR_UNSUPPORTED;
  if (M == 0) return FP_OK;
  size_t need = linear_ws_bytes(wquant, M, N, K);
  // quantised prefill without room for the bf16 expansion: the GEMM that
  // dequantises in the kernel needs no workspace
  const bool no_scratch = !workspace || workspace_bytes < need;
  const bool in_kernel = M > 64 && wquant != FP_W_BF16 && no_scratch && gemm_wq_ok(wquant, epilogue, M, N, K, x, codes);
  if (need > 0 && no_scratch && !in_kernel) return FP_ERR_INVALID_ARG;
  return cuda_status(launch_linear(wquant, epilogue, x, M, N, K, codes, scales, zeros, residual, y, workspace,
                                   workspace_bytes, (cudaStream_t)stream));
}

int fp_op_rmsnorm(const uint16_t* x, int M, int d, int row_stride, int row_offset, const uint16_t* g, float eps,
                  uint16_t* y, void* stream) {
  if (!x || !g || !y || M < 0 || d <= 0 || row_stride < 0 || row_offset < 0) return FP_ERR_INVALID_ARG;
  if (!(eps >= 0.f)) return FP_ERR_INVALID_ARG;
  if (d % 8 != 0) return FP_ERR_UNSUPPORTED;
  return cuda_status(launch_rmsnorm(x, M, d, row_stride, row_offset, g, eps, y, (cudaStream_t)stream));
}

int fp_op_embed(const int32_t* tok, int M, const uint16_t* E, int V, int d, uint16_t* h, int32_t* err,
                void* stream) {
  if (!tok || !E || !h || M < 0 || V <= 0 || d <= 0) return FP_ERR_INVALID_ARG;
  if (d % 8 != 0) return FP_ERR_UNSUPPORTED;
  return cuda_status(launch_embed(tok, M, E, V, d, h, err, (cudaStream_t)stream));
}

int fp_op_rope_table(int max_pos, int head_dim, float base, float* cs, void* stream) {
  if (max_pos <= 0 || head_dim <= 0 || head_dim % 2 != 0 || !(base > 0.f) || !cs) return FP_ERR_INVALID_ARG;
  const int half = head_dim / 2;
  std::vector<float> host((size_t)max_pos * half * 2);
  for (int p = 0; p < max_pos; ++p)
    for (int i = 0; i < half; ++i) {
      // theta_i = base^(-2i/hd), angle p * theta_i, in fp64 then rounded to fp32
      const double th = pow((double)base, -2.0 * (double)i / (double)head_dim);
      const double a = (double)p * th;
      host[((size_t)p * half + i) * 2 + 0] = (float)cos(a);
      host[((size_t)p * half + i) * 2 + 1] = (float)sin(a);
    }
  cudaError_t e = cudaMemcpyAsync(cs, host.data(), host.size() * sizeof(float), cudaMemcpyHostToDevice,
                                  (cudaStream_t)stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
  return cuda_status(e);
}

int fp_op_rope_kv(uint16_t* qkv, int B, int S, int row_stride, int n_heads, const fp_kv_view* kv,
                  const int32_t* pos, const float* rope_cs, int32_t* err, void* stream) {
  int st = fpk_check_kv(kv);
  if (st) return st;
  if (!qkv || !pos || !rope_cs || B < 0 || S < 0 || n_heads <= 0) return FP_ERR_INVALID_ARG;
  if (n_heads % kv->n_kv_heads != 0) return FP_ERR_INVALID_ARG;
  if (row_stride < (n_heads + 2 * kv->n_kv_heads) * kv->head_dim) return FP_ERR_INVALID_ARG;
  return cuda_status(launch_rope_kv(qkv, B, S, row_stride, n_heads, *kv, pos, rope_cs, err, (cudaStream_t)stream));
}

size_t fp_op_attention_decode_workspace_bytes(int B, int n_heads, int head_dim, int max_len) {
  if (B <= 0 || n_heads <= 0 || head_dim <= 0 || max_len <= 0) return 0;
  return attention_decode_ws_bytes(B, n_heads, head_dim, max_len);
}

int fp_op_attention_decode_splits(int B, int n_kv_heads, int head_dim, int kvquant, int max_len) {
  if (B <= 0 || n_kv_heads <= 0 || head_dim <= 0 || max_len <= 0) return 0;
  return attention_decode_splits(B, n_kv_heads, head_dim, kvquant, max_len);
}

static bool group_ok(int n_heads, int n_kv_heads) {
  if (n_heads % n_kv_heads != 0) return false;
  int G = n_heads / n_kv_heads;
  return G == 1 || G == 2 || G == 4 || G == 8;
}

int fp_op_attention_decode(const uint16_t* q, int q_stride, int B, int n_heads, const fp_kv_view* kv,
                           const int32_t* len, int max_len, uint16_t* out, void* workspace, size_t workspace_bytes,
                           int32_t* err, void* stream) {
  int st = fpk_check_kv(kv);
  if (st) return st;
  if (!q || !len || !out || B < 0 || n_heads <= 0 || max_len <= 0) return FP_ERR_INVALID_ARG;
  if (n_heads % kv->n_kv_heads != 0) return FP_ERR_INVALID_ARG;
  if (!group_ok(n_heads, kv->n_kv_heads)) return FP_ERR_UNSUPPORTED;
  if (q_stride < n_heads * kv->head_dim) return FP_ERR_INVALID_ARG;
  if (max_len > kv->pages_per_seq * kv->page_size) return FP_ERR_CAPACITY;
  if (B == 0) return FP_OK;
  if (!workspace || workspace_bytes < attention_decode_ws_bytes(B, n_heads, kv->head_dim, max_len))
    return FP_ERR_INVALID_ARG;
  return cuda_status(launch_attention_decode(q, q_stride, B, n_heads, *kv, len, 0, max_len, out, workspace, err,
                                             (cudaStream_t)stream));
}

int fp_op_attention_prefill(const uint16_t* q, int q_stride, int B, int S, int n_heads, const fp_kv_view* kv,
                            uint16_t* out, int32_t* err, void* stream) {
  int st = fpk_check_kv(kv);
  if (st) return st;
  if (!q || !out || B < 0 || S < 0 || n_heads <= 0) return FP_ERR_INVALID_ARG;
  if (n_heads % kv->n_kv_heads != 0) return FP_ERR_INVALID_ARG;
  if (q_stride < n_heads * kv->head_dim) return FP_ERR_INVALID_ARG;
  if (S > kv->pages_per_seq * kv->page_size) return FP_ERR_CAPACITY;
  return cuda_status(launch_attention_prefill(q, q_stride, B, S, n_heads, *kv, out, err, (cudaStream_t)stream));
}

int fp_op_argmax(const float* logits, int M, int V, int32_t* out, void* stream) {
  if (!logits || !out || M < 0 || V <= 0) return FP_ERR_INVALID_ARG;
  return cuda_status(launch_argmax(logits, M, V, out, (cudaStream_t)stream));
}

}  // extern "C"
