/*
 * fp.h -- C ABI of the GB300 fingerprint profiler.
 *
 * A fingerprint is an LLM rebuilt with the same components (embedding,
 * decoder blocks, linear layers, normalisation, activation, softmax) but one
 * or two hidden layers (arXiv 2501.13111, Sec. 1 "Our work" and Sec. 5.1).
 * Profiling deploys it under one configuration, sends dummy requests and
 * reads latency and memory (Sec. 4.2 step 1; Sec. 7 "Fingerprint
 * Controller"); the estimator then needs TTFT and TPOT (Eq. 1-3, Sec. 5.3)
 * and the footprint (Sec. 5.2).  This library runs that forward pass on one
 * GPU with its own CUDA kernels and reports those numbers.
 *
 * Conventions (every function):
 *   - Return FP_OK (0) on success or a negative FP_ERR_* code; the handle's
 *     message (fp_last_error) says why.  No function aborts the process.
 *   - Host pointers are borrowed for the duration of the call only.
 *   - The handle owns every device allocation it makes and frees them in
 *     fp_destroy.  With an fp_allocator, all of them go through it.
 *   - Work runs on the handle's stream.  A call returns before the GPU has
 *     finished unless it hands results back to host memory.
 *   - A handle must not be used from two threads at once.
 */
#ifndef FP_H
#define FP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ----------------------------------------------------------- status codes */
#define FP_OK                 0
#define FP_ERR_INVALID_ARG   -1  /* a NULL, negative, out-of-range or inconsistent argument */
#define FP_ERR_UNSUPPORTED   -2  /* a valid shape this build does not implement (see fp_create) */
#define FP_ERR_OOM           -3  /* an allocation failed (cudaMalloc or the caller's allocator) */
#define FP_ERR_CUDA          -4  /* a CUDA runtime call failed; no device, or a launch error */
#define FP_ERR_CAPACITY      -5  /* the KV cache has no room for the requested positions */
#define FP_ERR_DEVICE_ASSERT -6  /* a kernel found a bad index (token id, page) and skipped it */
#define FP_ERR_STATE         -7  /* call out of order, e.g. decode before any prefill */

/* ---------------------------------------------------------- configuration */
/* Weight-only quantisation of the block linear layers (Sec. 3.2; table
 * "Models and configurations").  Embedding, norm gains and LM head stay bf16.
 *   FP_W_BF16       : bf16 [N][K]
 *   FP_W_INT8       : int8 codes [N][K] + one bf16 scale per output row [N];
 *                     w = q * s, s = bf16 round-up of max|w_row| / 127
 *   FP_W_INT4_G128  : uint8 [N][K/2]: each little-endian 32-bit word holds
 *                     8 consecutive elements e0..e7 of a row, nibble i
 *                     (bits 4i..4i+3) = element (0,2,4,6,1,3,5,7)[i], so the
 *                     nibbles a 0x000F000F mask picks are a consecutive pair;
 *                     + bf16 scale and bf16 zero per row and 128-wide group
 *                     of K, [N][K/128] each; w = (q - z) * s
 *   FP_W_GPTQ4      : GPTQ-format int4 with act order ("GPTQ4" in the same
 *                     table): an act order perm, int32 [K], a permutation of
 *                     the input channels; group g holds the channels
 *                     perm[128g .. 128g+127] (GPTQ's g_idx[perm[j]] = j/128).
 *                     Codes, scales and zeros are the FP_W_INT4_G128 layout
 *                     of the matrix read in act order (stored column j is
 *                     channel perm[j]): w[n][perm[j]] = (q[n][j] - z[n][j/128])
 *                     * s[n][j/128].  Without calibration data the codes are
 *                     the int4 rule on each group's values (round to nearest).
 *                     fp_create draws one act order per fused matrix from the
 *                     seed (Fisher-Yates over SplitMix64).                  */
enum { FP_W_BF16 = 0, FP_W_INT8 = 1, FP_W_INT4_G128 = 2, FP_W_GPTQ4 = 3 };

/* KV cache format (INT8 KV cache: table "Models and configurations").
 *   FP_KV_BF16 : K and V as bf16
 *   FP_KV_INT8 : int8 codes + one fp32 scale per (token, KV head), separately
 *                for K (after RoPE) and V; s = max|x| / 127              */
enum { FP_KV_BF16 = 0, FP_KV_INT8 = 1 };

/* Decoder shape.  Block = pre-norm RMSNorm, rotate-half RoPE, grouped-query
 * attention (query head j reads KV head j / (n_heads / n_kv_heads)), SwiGLU
 * FFN, residual adds; then final RMSNorm and an untied LM head. */
typedef struct fp_arch {
  int n_layers;    /* decoder blocks, 1 .. FP_MAX_LAYERS                   */
  int hidden;      /* d                                                    */
  int n_heads;     /* query heads H                                        */
  int n_kv_heads;  /* KV heads Hkv, H % Hkv == 0                           */
  int head_dim;    /* hd, 64 or 128                                        */
  int ffn;         /* f, SwiGLU inner width                                */
  int vocab;       /* V                                                    */
  float rms_eps;   /* e.g. 1e-5                                            */
  float rope_base; /* e.g. 10000                                           */
} fp_arch;

#define FP_MAX_LAYERS 80 /* Llama-2-70B depth: the full model runs too */

/* Optional device allocator.  alloc returns a device pointer aligned to at
 * least 256 bytes, or NULL on failure (fp_create then returns FP_ERR_OOM and
 * frees what it already took).  free releases one pointer from alloc. */
typedef struct fp_allocator {
  void* (*alloc)(size_t bytes, void* ctx);
  void (*free)(void* ptr, void* ctx);
  void* ctx;
} fp_allocator;

/* fp_create flags */
#define FP_FLAG_KEEP_HIDDEN 1u /* keep each block's output for fp_get_tensor */
#define FP_FLAG_NO_INIT     2u /* skip the seeded weight fill (caller sets every tensor) */

typedef struct fp_handle fp_handle;

/* Create a fingerprint under one deployment configuration.
 *   batch       : sequences per request batch, >= 1
 *   max_context : KV capacity per sequence (prompt + generated), >= 1
 *   page_size   : tokens per KV page, 16 (the only size built)
 *   seed        : weights are drawn by SplitMix64 (counter-based) and an
 *                 Irwin-Hall(4) approximate N(0, 0.02), rounded to bf16,
 *                 then quantised; norm gains are 1.0
 *   flags       : FP_FLAG_*
 *   alloc       : NULL = cudaMalloc/cudaFree
 *   stream      : cudaStream_t; NULL = a stream the handle creates and owns
 * Shape limits (FP_ERR_UNSUPPORTED): head_dim not 64/128; hidden not a
 * multiple of 64 or ffn not a multiple of 32 (both multiples of 128 with int4
 * or GPTQ4 weights); page_size != 16; n_layers > FP_MAX_LAYERS.
 * All device memory (weights, KV pages, activations for a prefill of
 * batch * max_context tokens, workspaces) is reserved here once; that sum is
 * the peak footprint fp_profile reports. */
int fp_create(const fp_arch* arch, int wquant, int kvquant, int batch, int max_context,
              int page_size, unsigned long long seed, unsigned flags, const fp_allocator* alloc,
              void* stream, fp_handle** out);

/* Tensor ids for fp_set_weight.  layer >= 0: one decoder block; layer == -1:
 * the global tensors. */
enum {
  FP_T_ATTN_NORM = 0, /* [d]            */
  FP_T_WQ = 1,        /* [H*hd][d]      */
  FP_T_WK = 2,        /* [Hkv*hd][d]    */
  FP_T_WV = 3,        /* [Hkv*hd][d]    */
  FP_T_WO = 4,        /* [d][H*hd]      */
  FP_T_FFN_NORM = 5,  /* [d]            */
  FP_T_WGATE = 6,     /* [f][d]         */
  FP_T_WUP = 7,       /* [f][d]         */
  FP_T_WDOWN = 8      /* [d][f]         */
};
enum { FP_T_EMBED = 0 /* [V][d] */, FP_T_FINAL_NORM = 1 /* [d] */, FP_T_LM_HEAD = 2 /* [V][d] */ };

/* Replace one weight tensor with host bf16 values (uint16 bit patterns,
 * row-major, n_elems must equal the tensor's size) and re-quantise it into
 * the configuration's format on the GPU.  Synchronous. */
int fp_set_weight(fp_handle* h, int layer, int tensor, const uint16_t* host_bf16, size_t n_elems);

/* Set the page table: host int32 [batch][pages_per_seq] of physical page
 * ids, each in [0, batch * pages_per_seq) and used at most once
 * (FP_ERR_INVALID_ARG otherwise).  pages_per_seq = ceil(max_context / 16).
 * The default maps page p of sequence b to p * batch + b. */
int fp_set_page_table(fp_handle* h, const int32_t* host_table);

/* Load a prompt into the device-resident prompt buffer: host_tokens
 * [batch][prompt_len] (ids in [0, vocab)), or NULL for SplitMix64 ids drawn
 * from the handle's seed (stream 2^20, multiply-shift onto [0, vocab)).
 * Synchronous with respect to host_tokens. */
int fp_load_prompt(fp_handle* h, const int32_t* host_tokens, int prompt_len);

/* Prefill: run the prompt through the fingerprint from an empty cache, fill
 * the KV cache and emit the first generated token per sequence (greedy).
 * This is the dummy request of the profiling step (Sec. 4.2, step 1) up to
 * its first token: its duration is the TTFT of Eq. 1 (Sec. 5.3).
 * host_tokens [batch][prompt_len] is uploaded first; with host_tokens NULL
 * the resident prompt of fp_load_prompt is used (prompt_len must equal its
 * length, else FP_ERR_STATE).  host_next [batch] or NULL; with NULL the
 * tokens stay on the device for the next decode step. */
int fp_prefill(fp_handle* h, const int32_t* host_tokens, int prompt_len, int32_t* host_next);

/* One decode step: consume one token per sequence (host_in [batch], or NULL
 * for the previous step's outputs kept on the device), append one position,
 * emit the next greedy token (host_out [batch] or NULL).  One step is one
 * output token of Eq. 1 (Sec. 5.3); the KV cache makes every step cost the
 * same work per layer (the passage before Eq. 1), so its duration is TPOT.  FP_ERR_STATE
 * before any prefill; FP_ERR_CAPACITY when the cache is full.  The step is a
 * replayed CUDA graph (captured on first use). */
int fp_decode_step(fp_handle* h, const int32_t* host_in, int32_t* host_out);

/* n decode steps that feed their own tokens back, all on the device
 * (n graph replays, nothing crosses the host boundary; asynchronous). */
int fp_decode_steps(fp_handle* h, int n);

/* Kernel classes timed by fp_profile.  FP_K_EMBED is the embedding gather
 * fused with the first block's pre-attention RMSNorm; FP_K_ARGMAX also moves
 * every sequence's position past the pass. */
enum {
  FP_K_EMBED = 0, FP_K_RMSNORM, FP_K_LIN_QKV, FP_K_ROPE_KV, FP_K_ATTN, FP_K_ATTN_COMBINE,
  FP_K_LIN_O, FP_K_LIN_GU, FP_K_LIN_DOWN, FP_K_LM_HEAD, FP_K_ARGMAX, FP_K_COUNT
};

typedef struct fp_profile_result {
  double ttft_ms;             /* prefill to first token, device events, mean over iters */
  double tpot_ms;             /* mean decode step (graph replay)                  */
  double tpot_ms_p50;         /* median decode step                               */
  double decode_tokens_per_s; /* batch * n_decode / total decode time             */
  double prefill_tflops;      /* prefill_flops / ttft                             */
  double prefill_flops;       /* algorithmic, oracle/memory.py formula            */
  double block_ms[FP_MAX_LAYERS]; /* per block, mean per decode step (eager pass with events) */
  double other_ms;            /* embedding + final norm + LM head + argmax per step */
  double kernel_ms[FP_K_COUNT];   /* per class, summed over the step, mean per step;
                                     FP_K_ATTN includes its combine kernel        */
  int kernel_launches[FP_K_COUNT];/* timed intervals per decode step, per class     */
  int decode_launches;            /* kernels one decode step launches             */
  int prefill_launches;           /* kernels one prefill launches                 */
  unsigned long long block_bytes[FP_MAX_LAYERS]; /* algorithmic bytes of block l at the mean context */
  unsigned long long peak_hbm_bytes;   /* everything the handle reserved           */
  unsigned long long weight_bytes, kv_bytes, act_bytes, workspace_bytes;
  unsigned long long memgetinfo_bytes; /* cudaMemGetInfo drop across fp_create    */
  unsigned long long decode_bytes_per_step; /* algorithmic, at the mean context   */
  int n_layers, prompt_len, n_decode, iters;
  double request_ms;          /* one request: prefill + n_decode decode steps, device
                                 events, mean over iters (the latency of Eq. 1) */
  unsigned long long observed_hbm_bytes; /* device memory the deployment holds at the end
                                 of fp_profile: free memory just before fp_create minus
                                 free memory now (cudaMemGetInfo), the reading a monitor of
                                 the GPU takes (Sec. 7 "Monitoring Daemon"); it counts
                                 whatever else the process allocated in between */
} fp_profile_result;

/* Profile latency and memory, the observations the estimator consumes:
 * TTFT and TPOT of Eq. 1 (Sec. 5.3; with two fingerprint depths, Eqs. 2-3
 * separate their per-layer and other parts) and the footprint W + A of the
 * memory model (Sec. 5.2, TP = PP = 1), as the profiling step reads them
 * from a deployed fingerprint (Sec. 4.2, step 1; Sec. 7 "Monitoring
 * Daemon").  `warmup` untimed passes, then `iters` timed
 * passes of prefill(prompt_len) + n_decode decode steps on the batch;
 * prompt = host_prompt [batch][prompt_len] or, if NULL, SplitMix64 token ids
 * drawn from the handle's seed.  prompt_len + n_decode <= max_context. */
int fp_profile(fp_handle* h, int prompt_len, int n_decode, int warmup, int iters,
               const int32_t* host_prompt, fp_profile_result* out);

/* Reads for tests (synchronous).  Returns bytes written, or the size needed
 * when host_dst is NULL, or an FP_ERR_* code.  A host buffer smaller than the
 * tensor receives its leading `bytes` bytes (e.g. the first rows of
 * FP_G_HIDDEN, which are sequence 0's).  `mat` picks a fused matrix:
 * FP_M_QKV = [Wq; Wk; Wv], FP_M_O, FP_M_GU = [Wgate; Wup], FP_M_DOWN. */
enum { FP_M_QKV = 0, FP_M_O = 1, FP_M_GU = 2, FP_M_DOWN = 3 };
enum {
  FP_G_W_CODES = 0,  /* (layer, mat) codes as stored                             */
  FP_G_W_SCALES = 1, /* (layer, mat) bf16 scales                                 */
  FP_G_W_ZEROS = 2,  /* (layer, mat) bf16 zeros (int4)                           */
  FP_G_K_POOL = 3,   /* (layer) whole K page pool [pages][Hkv][16][hd]           */
  FP_G_V_POOL = 4,
  FP_G_K_SCALES = 5, /* (layer) fp32 [pages][Hkv][16] (int8 KV)                  */
  FP_G_V_SCALES = 6,
  FP_G_HIDDEN = 7,   /* (layer) block output of the last call, bf16 [rows][d]   */
  FP_G_LOGITS = 8,   /* fp32 [batch][vocab] of the last call                     */
  FP_G_TOKENS = 9,   /* int32 [batch] last emitted tokens                        */
  FP_G_PAGE_TABLE = 10, /* int32 [batch][pages_per_seq]                          */
  FP_G_LENGTH = 11,  /* int32 [batch] cached positions per sequence              */
  FP_G_W_PERM = 12   /* (layer, mat) int32 [K] act order of a GPTQ4 matrix         */
};
long long fp_get_tensor(fp_handle* h, int what, int layer, int mat, void* host_dst, size_t bytes);

/* As fp_get_tensor, from byte `offset` of the tensor on: returns the bytes
 * written, or (host_dst NULL) the bytes from offset to the end; an offset
 * past the end is FP_ERR_INVALID_ARG.  Lets a test read one sequence's rows
 * of FP_G_HIDDEN (sequence b starts at b * rows_per_sequence * d * 2). */
long long fp_get_tensor_at(fp_handle* h, int what, int layer, int mat, size_t offset, void* host_dst,
                           size_t bytes);

/* Byte plan of the handle (what fp_profile reports as peak_hbm_bytes). */
typedef struct fp_plan {
  unsigned long long weight_bytes, kv_bytes, act_bytes, workspace_bytes, total_bytes;
  int pages_per_seq, max_rows;
} fp_plan;
int fp_get_plan(const fp_handle* h, fp_plan* out);

const char* fp_last_error(const fp_handle* h);
const char* fp_strerror(int code);
void fp_destroy(fp_handle* h);

#ifdef __cplusplus
}
#endif
#endif /* FP_H */
