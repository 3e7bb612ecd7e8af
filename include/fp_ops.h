/*
 * fp_ops.h -- one C entry point per step of the fingerprint forward pass.
 *
 * These are the kernels the fingerprint runtime (fp.h) strings together,
 * exposed one by one on caller-owned DEVICE buffers so each step can be
 * checked against the oracle and timed alone.  Steps follow the decoder
 * block the fingerprint keeps from its LLM (arXiv 2501.13111, Sec. 1 "Our
 * work", Sec. 5.1) under the deployment configurations of Sec. 3.2 (weight
 * and KV-cache quantisation).
 *
 * Conventions:
 *   - Every pointer argument is a device pointer unless its name starts
 *     with host_.  Buffers are row-major; bf16 is passed as its uint16 bits.
 *   - The launch is asynchronous on `stream` (cudaStream_t, NULL = legacy
 *     default stream).  Arguments are checked on the host before any launch:
 *     FP_ERR_INVALID_ARG / FP_ERR_UNSUPPORTED and nothing is launched.
 *     FP_ERR_CUDA if the launch itself fails.  Nothing is allocated.
 *   - Output buffers must not overlap inputs unless a function says so.
 *   - Return codes are the FP_* codes of fp.h.
 */
#ifndef FP_OPS_H
#define FP_OPS_H

#include <stddef.h>
#include <stdint.h>

#include "fp.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Quantise a bf16 weight matrix w [N][K] into the wquant format of fp.h
 * (Sec. 3.2; formats in fp.h).  int8: codes int8 [N][K], scales bf16 [N].
 * int4: codes uint8 [N][K/2], scales and zeros bf16 [N][K/128]; K % 128 == 0.
 * bf16: codes receives a copy of w.  Codes are bit-exact with the reading
 * (fp32 IEEE division, round half to even). */
int fp_op_quantize(int wquant, const uint16_t* w, int N, int K, void* codes, uint16_t* scales,
                   uint16_t* zeros, void* stream);

/* Quantise w [N][K] (bf16) into the FP_W_GPTQ4 format of fp.h: int4 over
 * the act-order groups of perm (int32 [K], a permutation of 0..K-1; group g
 * holds the channels perm[128g .. 128g+127]), codes stored in act order
 * ([N][K/2], the int4 packing), scales and zeros bf16 [N][K/128]
 * (GPTQ4, Sec. 3.2 and the table "Models and configurations").  K % 128 ==
 * 0.  An entry of perm outside [0, K) reads as a zero weight. */
int fp_op_quantize_gptq4(const uint16_t* w, int N, int K, const int32_t* perm, void* codes, uint16_t* scales,
                         uint16_t* zeros, void* stream);

/* Fill w [n] with the seeded bf16 weights of stream `stream_id` (SplitMix64
 * counter-based draws, Irwin-Hall(4), sigma 0.02; elements start..start+n-1). */
int fp_op_init_weights(uint16_t* w, long long n, unsigned long long seed, long long stream_id,
                       long long start, void* stream);

/* Epilogues of fp_op_linear. */
enum {
  FP_EPI_STORE = 0,  /* y bf16 [M][N]                                          */
  FP_EPI_RESID = 1,  /* y bf16 [M][N] = residual + x W^T; residual may equal y  */
  FP_EPI_SWIGLU = 2, /* W rows = [gate (N/2 rows); up (N/2 rows)];
                        y bf16 [M][N/2] = silu(x Wg^T) * (x Wu^T)             */
  FP_EPI_F32 = 3     /* y fp32 [M][N]                                          */
};

/* Weight-only linear y = x W^T (the "linear layers" of the block) with the
 * dequantisation fused: x bf16 [M][K]; W in the wquant format of fp.h
 * (codes / scales / zeros as fp_op_quantize writes them); fp32 accumulation.
 * Kernel choice depends on M, N and K: M <= 64 runs the decode GEMV (the
 * work is cut into equal ranges of (128-row block, K step), one per resident
 * CTA, and shared blocks are reduced from fp32 partials in a fixed order) --
 * on mma.sync with the codes dequantised in registers, except, with 16-byte
 * aligned x and codes: int4 with 17 <= M <= 64 (K a multiple of 128), and
 * int8 with 33 <= M <= 64 or K >= 16384, which run on tcgen05 with each
 * weight expanded in TMEM (int4 to bf16((q - z) s) as the prefill GEMM does,
 * int8 to the integer code, its row scale applied to the fp32 sums); bf16
 * with 17 <= M <= 64 on matrices that give every SM at least 48 items of 32
 * KB, which runs on tcgen05 fed by TMA; a K that is not a multiple of the
 * GEMV's K step falls back to one warp per output row on the CUDA cores --
 * larger M the tcgen05 GEMM.  For M > 64 with int8
 * or int4 weights the GEMM either reads a bf16 expansion of W that it writes
 * into the workspace band by band (at most 128 MB; the faster path), or, when
 * the workspace is NULL or smaller than that, dequantises the codes inside
 * the GEMM (bf16 weight tiles built in shared memory for every 256-token
 * tile; no workspace; about two thirds of the speed; x and codes 16-byte
 * aligned).  workspace: 16-byte aligned, at least
 * fp_op_linear_workspace_bytes(wquant, M, N, K) bytes (may be NULL when that
 * is 0, or for the in-kernel dequantisation above), else FP_ERR_INVALID_ARG.
 * Its leading bytes are ticket counters
 * that must be zero before the first call (e.g. a zeroed buffer); every call
 * leaves them zero again, so one workspace serves any sequence of calls on
 * one stream (calls that overlap on the GPU need separate workspaces). */
int fp_op_linear(int wquant, int epilogue, const uint16_t* x, int M, int N, int K, const void* codes,
                 const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                 void* workspace, size_t workspace_bytes, void* stream);
size_t fp_op_linear_workspace_bytes(int wquant, int M, int N, int K);

/* The weight-only linear of fp_op_linear for FP_W_GPTQ4 weights (codes,
 * scales, zeros as fp_op_quantize_gptq4 writes them; perm the act order).
 * y = x W^T with W in channel order.  M <= 64: x is gathered into the act
 * order in the workspace (one kernel) and the int4 decode linear runs on it;
 * M > 64: the weights are expanded back into channel order (the inverse act
 * order is computed into the workspace) and the prefill GEMM multiplies x as
 * it is.  workspace: 256-byte aligned, at least
 * fp_op_linear_gptq4_workspace_bytes(M, N, K) bytes, its leading ticket
 * counters zero before the first call (every call leaves them zero).  An
 * entry of perm outside [0, K) reads as zero and sets *err = 1 (err may be
 * NULL).  K % 128 == 0 (FP_ERR_UNSUPPORTED). */
int fp_op_linear_gptq4(int epilogue, const uint16_t* x, int M, int N, int K, const int32_t* perm, const void* codes,
                       const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                       void* workspace, size_t workspace_bytes, int32_t* err, void* stream);
size_t fp_op_linear_gptq4_workspace_bytes(int M, int N, int K);

/* RMSNorm of selected rows: y[r] = x[r*row_stride + row_offset] /
 * sqrt(mean(x^2) + eps) * g, r < M; x, y, g bf16; fp32 arithmetic. */
int fp_op_rmsnorm(const uint16_t* x, int M, int d, int row_stride, int row_offset, const uint16_t* g,
                  float eps, uint16_t* y, void* stream);

/* Embedding gather h[m] = E[tok[m]]; tok int32 [M], E bf16 [V][d].  An id
 * outside [0, V) writes a zero row and sets *err = 1 (err may be NULL). */
int fp_op_embed(const int32_t* tok, int M, const uint16_t* E, int V, int d, uint16_t* h, int32_t* err,
                void* stream);

/* Paged KV cache view.  Pools are [n_pages][n_kv_heads][page_size][head_dim]
 * (bf16 or int8 codes); scales (int8 only) fp32 [n_pages][n_kv_heads][page_size];
 * page_table int32 [batch][pages_per_seq]: position p of sequence b lives in
 * page page_table[b][p / page_size], slot p % page_size. */
typedef struct fp_kv_view {
  int kvquant, n_kv_heads, head_dim, page_size, pages_per_seq, n_pages;
  void* k_pool;
  void* v_pool;
  float* k_scale;
  float* v_scale;
  const int32_t* page_table;
} fp_kv_view;

/* RoPE table for positions 0..max_pos-1: cs fp32 [max_pos][head_dim/2][2] =
 * (cos, sin) of p * base^(-2i/hd), computed on the host in fp64 and rounded
 * to fp32, then copied to the device (synchronous). */
int fp_op_rope_table(int max_pos, int head_dim, float base, float* cs, void* stream);

/* RoPE + KV-cache append.  qkv bf16 [B*S][row_stride]: per token, H query
 * heads, then Hkv key heads, then Hkv value heads, head_dim each.  Token s
 * of sequence b sits at position pos[b] + s.  Query and key heads are
 * rotated (rotate-half); queries are written back in place; keys (rotated,
 * rounded to bf16) and values go to the cache, quantised per (token, KV
 * head) when kvquant is int8.  rope_cs (fp_op_rope_table) must cover
 * pages_per_seq * page_size positions.  A position outside
 * [0, pages_per_seq * page_size) or a page id outside the pool sets
 * *err = 1 (err may be NULL) and skips that head. */
int fp_op_rope_kv(uint16_t* qkv, int B, int S, int row_stride, int n_heads, const fp_kv_view* kv,
                  const int32_t* pos, const float* rope_cs, int32_t* err, void* stream);

/* Decode attention: one query row per sequence, q bf16 [B][q_stride] (head h
 * at h*head_dim), attends over positions 0 .. len[b]-1 of the cache
 * (softmax(q K^T / sqrt(hd)) V, query head j reads KV head j / (H/Hkv));
 * out bf16 [B][n_heads*head_dim].  Split over the context in chunks; the
 * partial results go to `workspace` (fp_op_attention_decode_workspace_bytes
 * for at most max_len cached positions) and a second kernel combines them.
 * len[b] in [1, max_len]; a larger len[b] is clipped to max_len and sets
 * *err = 1 (err may be NULL). */
int fp_op_attention_decode(const uint16_t* q, int q_stride, int B, int n_heads, const fp_kv_view* kv,
                           const int32_t* len, int max_len, uint16_t* out, void* workspace,
                           size_t workspace_bytes, int32_t* err, void* stream);
size_t fp_op_attention_decode_workspace_bytes(int B, int n_heads, int head_dim, int max_len);

/* Context splits fp_op_attention_decode uses for B sequences, n_kv_heads KV
 * heads of head_dim, a kvquant cache of 16-token pages with 16-byte aligned
 * pools, and max_len cached positions (0 for a non-positive argument).  With
 * 1 split the kernel normalises in place and never touches the workspace;
 * with more, the partials go to the workspace and a second kernel merges
 * them. */
int fp_op_attention_decode_splits(int B, int n_kv_heads, int head_dim, int kvquant, int max_len);

/* Decode attention without a caller workspace, for callers that cannot
 * allocate device memory (a host whose device memory is all reserved by
 * another framework's pool, a plugin that must not call the allocator, a
 * latency-critical loop that cannot risk the synchronisation of cudaMalloc).
 * The paper has no counterpart: this is a deployment convenience of this
 * library only.
 *
 * Same arguments, kernels and results as fp_op_attention_decode, but the
 * split partials go to a scratch array of FP_NOALLOC_SCRATCH_BYTES (32 MiB)
 * compiled into the library.  Every GPU that loads the library holds that
 * array until the process exits.  The call allocates nothing.
 *   - A request whose fp_op_attention_decode_workspace_bytes(B, n_heads,
 *     head_dim, max_len) exceeds FP_NOALLOC_SCRATCH_BYTES returns
 *     FP_ERR_UNSUPPORTED before anything is launched.
 *   - The first call on a device looks up the array's device address on that
 *     device (cudaGetSymbolAddress, with the device current) and caches it
 *     with the id of the device's current context; make that first call
 *     before any stream capture.  After a device reset the context differs,
 *     and the next call looks the address up again (make it, too, outside a
 *     capture).
 *   - All calls share the one array, which keeps the last call's contents;
 *     each call writes every partial it reads back, so nothing needs
 *     clearing.  Calls that overlap on the GPU (other streams, other host
 *     threads) race on the array: serialise them. */
#define FP_NOALLOC_SCRATCH_BYTES (32u << 20)
int fp_op_attention_decode_noalloc(const uint16_t* q, int q_stride, int B, int n_heads, const fp_kv_view* kv,
                                   const int32_t* len, int max_len, uint16_t* out, int32_t* err, void* stream);

/* Prefill attention: causal, S query rows per sequence at positions 0..S-1,
 * q bf16 [B*S][q_stride]; keys/values read from the cache positions 0..S-1;
 * out bf16 [B*S][n_heads*head_dim].  head_dim 128 with 16-token pages,
 * 16-byte aligned q (q_stride a multiple of 8) and pools runs on tcgen05
 * (scores and output accumulated in TMEM); other shapes on mma.sync.  An
 * int8 cache enters as its codes, with each key's K scale multiplying its
 * score column and its V scale its probability column in fp32; on tcgen05
 * the int8-cache products run in fp16 (codes exact, q converted, P carrying
 * the V scales times a power of two that keeps it in the fp16 normal
 * range), and a q element beyond the fp16 range sets *err = 3 (the output
 * is then invalid).  A page id outside [0, n_pages) reads zeros and sets
 * *err = 1. */
int fp_op_attention_prefill(const uint16_t* q, int q_stride, int B, int S, int n_heads,
                            const fp_kv_view* kv, uint16_t* out, int32_t* err, void* stream);

/* Test hook for the failure path of the pipelined tensor-core kernels (the
 * paper has no counterpart).  Every wait of those kernels is bounded; a role
 * whose wait runs out stops, the CTA drains its copies and MMAs in flight,
 * frees its tensor memory and records status 2 in the error word, which the
 * runtime reports as FP_ERR_DEVICE_ASSERT.  This sets how many polling rounds
 * the prefill GEMM's MMA thread waits for a stage of operands on the current
 * device: rounds >= 0 (0 gives up at once) or < 0 to restore the default;
 * all other waits keep the default.  Synchronous; not for use while kernels
 * of the library are running. */
int fp_debug_set_wait_limit(long long rounds);

/* Greedy choice out[m] = argmax logits[m][:V] (fp32); ties to the lowest id. */
int fp_op_argmax(const float* logits, int M, int V, int32_t* out, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* FP_OPS_H */
