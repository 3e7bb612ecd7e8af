// Fingerprint runtime behind fp.h: byte plan and arena, seeded weights,
// paged KV cache, the prefill / decode kernel sequence, the decode CUDA graph
// and device-timed profiling.
//
// Profiling a fingerprint means deploying it under one configuration,
// sending dummy requests and reading latency and memory (Sec. 4.2 step 1;
// Sec. 7 "Fingerprint Controller").  Latency is reported as TTFT and TPOT
// (Eq. 1, Sec. 5.3) and memory as the bytes the deployment holds (W + A,
// Sec. 5.2).
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <string>
#include <vector>

#include "common.cuh"
#include "kernels.cuh"

using namespace fpk;

extern int fpk_check_kv(const fp_kv_view* kv);

namespace fpk {
thread_local bool g_pdl = false;
}

namespace {

thread_local std::string g_create_error;

struct Mat {
  void* codes = nullptr;
  uint16_t* scales = nullptr;
  uint16_t* zeros = nullptr;
  int32_t* perm = nullptr;  // GPTQ4: the act order [K] and its inverse
  int32_t* inv = nullptr;
  int N = 0, K = 0;
};

struct Layer {
  uint16_t* attn_norm = nullptr;
  uint16_t* ffn_norm = nullptr;
  Mat mat[4];  // FP_M_QKV, FP_M_O, FP_M_GU, FP_M_DOWN
  void* kpool = nullptr;
  void* vpool = nullptr;
  float* kscale = nullptr;
  float* vscale = nullptr;
};

// GPTQ4 stores an int4 g128 matrix (of the act-order channels) plus its act order
bool grouped(int wq) { return wq == FP_W_INT4_G128 || wq == FP_W_GPTQ4; }
size_t codes_bytes(int wq, long long N, long long K) {
  return wq == FP_W_BF16 ? N * K * 2 : wq == FP_W_INT8 ? N * K : N * K / 2;
}
size_t scale_bytes(int wq, long long N, long long K) {
  return wq == FP_W_BF16 ? 0 : wq == FP_W_INT8 ? N * 2 : N * (K / 128) * 2;
}
size_t zero_bytes(int wq, long long N, long long K) { return grouped(wq) ? N * (K / 128) * 2 : 0; }
size_t perm_bytes(int wq, long long K) { return wq == FP_W_GPTQ4 ? K * 4 : 0; }

// The act order of fused matrix m of block l: Fisher-Yates (Durstenfeld) over
// the identity, swapping entry i = K-1 .. 1 with the multiply-shift of draw
// K-1-i of stream (l + 1) * 16 + 9 + m onto [0, i] -- the definition the
// input generators of the tests implement too.
void act_order(unsigned long long seed, int l, int m, int K, int32_t* p) {
  for (int j = 0; j < K; ++j) p[j] = j;
  const uint64_t key = stream_key(seed, (uint64_t)(l + 1) * 16 + 9 + m);
  for (int t = 0; t + 1 < K; ++t) {
    const int i = K - 1 - t;
    const uint64_t hi = mix64(key + (uint64_t)(t + 1) * kGamma) >> 32;
    const int j = (int)((hi * (uint64_t)(i + 1)) >> 32);
    std::swap(p[i], p[j]);
  }
}

// Kernel-boundary event recorder for the instrumented (eager) decode pass.
struct Tracer {
  bool on = false;
  cudaStream_t s = nullptr;
  std::vector<cudaEvent_t> ev;
  std::vector<int> cls;  // class of the kernel that ends at ev[i] (i >= 1)
  std::vector<int> mark; // event index at block boundaries
  void start() {
    if (!on) return;
    push(-1);
  }
  void push(int c) {
    cudaEvent_t e;
    cudaEventCreate(&e);
    cudaEventRecord(e, s);
    ev.push_back(e);
    cls.push_back(c);
  }
  void after(int c) {
    if (on) push(c);
  }
  void boundary() {
    if (on) mark.push_back((int)ev.size() - 1);
  }
  void clear() {
    for (auto e : ev) cudaEventDestroy(e);
    ev.clear();
    cls.clear();
    mark.clear();
  }
};

}  // namespace

struct fp_handle {
  fp_arch a{};
  int wq = 0, kvq = 0, B = 0, T = 0, P = 16, pps = 0, n_pages = 0;
  unsigned long long seed = 0;
  unsigned flags = 0;
  fp_allocator alloc{};
  bool has_alloc = false;
  cudaStream_t stream = nullptr;
  bool own_stream = false;

  void* arena = nullptr;
  size_t arena_bytes = 0;
  unsigned long long weight_bytes = 0, kv_bytes = 0, act_bytes = 0, ws_bytes = 0, memgetinfo_bytes = 0;
  size_t free_before = 0;  // free device memory just before fp_create reserved anything

  uint16_t *embed = nullptr, *final_norm = nullptr, *lm_head = nullptr;
  Layer L[FP_MAX_LAYERS];
  int32_t *page_table = nullptr, *pos = nullptr, *tokens = nullptr, *prompt = nullptr, *err = nullptr;
  float* rope_cs = nullptr;
  uint16_t *h = nullptr, *y = nullptr, *qkv = nullptr, *att = nullptr, *act = nullptr, *ylast = nullptr;
  float* logits = nullptr;
  void* attn_ws = nullptr;
  size_t attn_ws_bytes = 0;
  void* lin_ws = nullptr;
  size_t lin_ws_bytes = 0;
  uint16_t* hidden = nullptr;  // [n_layers][max_rows][d]
  int max_rows = 0, n_qkv = 0, q_dim = 0;

  int length = 0;     // cached positions per sequence
  int last_rows = 0;  // rows of the last forward (hidden export)
  int launches = 0;   // kernels launched by the last forward
  int prefill_launches = 0;
  int prompt_len = 0; // length of the resident prompt (0 = none)
  bool prefilled = false;
  cudaGraphExec_t decode_exec = nullptr;
  Tracer tr;
  std::string msg;

  int fail(int code, const std::string& m) {
    msg = m;
    return code;
  }
  int cuda_fail(cudaError_t e, const char* where) {
    msg = std::string(where) + ": " + cudaGetErrorString(e);
    return FP_ERR_CUDA;
  }
  void* dev_alloc(size_t bytes) {
    if (has_alloc) return alloc.alloc(bytes, alloc.ctx);
    void* p = nullptr;
    return cudaMalloc(&p, bytes) == cudaSuccess ? p : nullptr;
  }
  void dev_free(void* p) {
    if (!p) return;
    if (has_alloc) alloc.free(p, alloc.ctx);
    else cudaFree(p);
  }
  fp_kv_view kv(int l) const {
    fp_kv_view v;
    v.kvquant = kvq;
    v.n_kv_heads = a.n_kv_heads;
    v.head_dim = a.head_dim;
    v.page_size = P;
    v.pages_per_seq = pps;
    v.n_pages = n_pages;
    v.k_pool = L[l].kpool;
    v.v_pool = L[l].vpool;
    v.k_scale = L[l].kscale;
    v.v_scale = L[l].vscale;
    v.page_table = page_table;
    return v;
  }
};

namespace {

// ---------------------------------------------------------------- byte plan
// Carves every device buffer out of one arena (256-byte aligned pieces).
// Called once with base = nullptr to size the arena, then with the arena.
struct Carver {
  char* base;
  size_t off = 0;
  template <class T>
  T* take(size_t bytes, unsigned long long* cat, unsigned long long exact = ~0ull) {
    size_t o = off;
    off += (bytes + 255) / 256 * 256;
    if (cat) *cat += exact == ~0ull ? bytes : exact;
    return base ? reinterpret_cast<T*>(base + o) : nullptr;
  }
};

void carve(fp_handle* h, char* base) {
  Carver c{base};
  const fp_arch& a = h->a;
  const long long d = a.hidden, f = a.ffn, V = a.vocab;
  h->weight_bytes = h->kv_bytes = h->act_bytes = h->ws_bytes = 0;
  h->embed = c.take<uint16_t>(V * d * 2, &h->weight_bytes);
  h->final_norm = c.take<uint16_t>(d * 2, &h->weight_bytes);
  h->lm_head = c.take<uint16_t>(V * d * 2, &h->weight_bytes);
  const int NK[4][2] = {{h->n_qkv, (int)d}, {(int)d, h->q_dim}, {(int)(2 * f), (int)d}, {(int)d, (int)f}};
  const size_t kv_elt = h->kvq == FP_KV_BF16 ? 2 : 1;
  const size_t pool = (size_t)h->n_pages * a.n_kv_heads * h->P * a.head_dim * kv_elt;
  const size_t spool = (size_t)h->n_pages * a.n_kv_heads * h->P * sizeof(float);
  for (int l = 0; l < a.n_layers; ++l) {
    Layer& L = h->L[l];
    L.attn_norm = c.take<uint16_t>(d * 2, &h->weight_bytes);
    L.ffn_norm = c.take<uint16_t>(d * 2, &h->weight_bytes);
    for (int m = 0; m < 4; ++m) {
      Mat& M = L.mat[m];
      M.N = NK[m][0];
      M.K = NK[m][1];
      M.codes = c.take<void>(codes_bytes(h->wq, M.N, M.K), &h->weight_bytes);
      size_t sb = scale_bytes(h->wq, M.N, M.K), zb = zero_bytes(h->wq, M.N, M.K);
      M.scales = sb ? c.take<uint16_t>(sb, &h->weight_bytes) : nullptr;
      M.zeros = zb ? c.take<uint16_t>(zb, &h->weight_bytes) : nullptr;
      // the act order is part of the stored matrix; its inverse only serves the prefill expansion
      M.perm = h->wq == FP_W_GPTQ4 ? c.take<int32_t>(perm_bytes(h->wq, M.K), &h->weight_bytes) : nullptr;
      M.inv = h->wq == FP_W_GPTQ4 ? c.take<int32_t>(perm_bytes(h->wq, M.K), &h->ws_bytes) : nullptr;
    }
    L.kpool = c.take<void>(pool, &h->kv_bytes);
    L.vpool = c.take<void>(pool, &h->kv_bytes);
    if (h->kvq == FP_KV_INT8) {
      L.kscale = c.take<float>(spool, &h->kv_bytes);
      L.vscale = c.take<float>(spool, &h->kv_bytes);
    } else {
      L.kscale = L.vscale = nullptr;
    }
  }
  h->page_table = c.take<int32_t>((size_t)h->B * h->pps * 4, &h->kv_bytes);
  const long long R = h->max_rows;
  h->pos = c.take<int32_t>(h->B * 4, &h->act_bytes);
  h->tokens = c.take<int32_t>(h->B * 4, &h->act_bytes);
  h->prompt = c.take<int32_t>((size_t)R * 4, &h->act_bytes);
  h->rope_cs = c.take<float>((size_t)h->pps * h->P * a.head_dim * sizeof(float), &h->act_bytes);
  h->h = c.take<uint16_t>(R * d * 2, &h->act_bytes);
  h->y = c.take<uint16_t>(R * d * 2, &h->act_bytes);
  h->qkv = c.take<uint16_t>(R * h->n_qkv * 2, &h->act_bytes);
  h->att = c.take<uint16_t>(R * h->q_dim * 2, &h->act_bytes);
  h->act = c.take<uint16_t>(R * f * 2, &h->act_bytes);
  h->ylast = c.take<uint16_t>(h->B * d * 2, &h->act_bytes);
  h->logits = c.take<float>((size_t)h->B * V * 4, &h->act_bytes);
  h->attn_ws_bytes = attention_decode_ws_bytes(h->B, a.n_heads, a.head_dim, h->T);
  h->attn_ws = c.take<void>(h->attn_ws_bytes, &h->ws_bytes);
  // every row count a forward can use: B (decode, LM head) and B * S for any prompt S
  size_t lw = 0;
  for (int m = 0; m < 4; ++m)
    lw = std::max(lw, h->wq == FP_W_GPTQ4 ? linear_gptq4_ws_bytes_upto((int)R, NK[m][0], NK[m][1], false)
                                          : linear_ws_bytes_upto(h->wq, (int)R, NK[m][0], NK[m][1]));
  lw = std::max(lw, linear_ws_bytes_upto(FP_W_BF16, h->B, (int)V, (int)d));
  h->lin_ws_bytes = lw;
  h->lin_ws = lw ? c.take<void>(lw, &h->ws_bytes) : nullptr;
  h->err = c.take<int32_t>(4, &h->ws_bytes);
  h->hidden = (h->flags & FP_FLAG_KEEP_HIDDEN) ? c.take<uint16_t>((size_t)a.n_layers * R * d * 2, &h->ws_bytes)
                                               : nullptr;
  h->arena_bytes = c.off;
}

bool bad_shape(const fp_arch* a, int wq, std::string& why) {
  char buf[200];
  if (a->head_dim != 64 && a->head_dim != 128) {
    snprintf(buf, sizeof buf, "head_dim %d: only 64 and 128 are built", a->head_dim);
    why = buf;
    return true;
  }
  int hm = grouped(wq) ? 128 : 64, fm = grouped(wq) ? 128 : 32;
  if (a->hidden % hm || a->ffn % fm || (a->n_heads * a->head_dim) % hm) {
    snprintf(buf, sizeof buf, "hidden %d / ffn %d / heads*head_dim %d not multiples of %d / %d / %d",
             a->hidden, a->ffn, a->n_heads * a->head_dim, hm, fm, hm);
    why = buf;
    return true;
  }
  int G = a->n_heads / a->n_kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8) {
    why = "n_heads / n_kv_heads must be 1, 2, 4 or 8";
    return true;
  }
  return false;
}

// ---------------------------------------------------------------- launches
#define LTRY(expr, cls)                                        \
  do {                                                         \
    cudaError_t e__ = (expr);                                  \
    if (e__ != cudaSuccess) return h->cuda_fail(e__, #cls);    \
    h->launches += 1;                                          \
    h->tr.after(cls);                                          \
  } while (0)

// One block linear: the GPTQ4 path (its decode gather counts as a launch of
// its own) or the weight-only linear of the handle's format.
cudaError_t block_linear(fp_handle* h, int epi, const uint16_t* x, int M, const Mat& W, const uint16_t* R, void* y) {
  if (h->wq == FP_W_GPTQ4) {
    if (M <= 64) h->launches += 1;
    return launch_linear_gptq4(epi, x, M, W.N, W.K, W.perm, W.inv, W.codes, W.scales, W.zeros, R, y, h->lin_ws,
                               h->lin_ws_bytes, h->stream, h->err);
  }
  return launch_linear(h->wq, epi, x, M, W.N, W.K, W.codes, W.scales, W.zeros, R, y, h->lin_ws, h->lin_ws_bytes,
                       h->stream, h->err);
}

// One forward pass over M = B * S rows (S tokens per sequence at positions
// pos[b] .. pos[b] + S - 1); tok: device ids [M].  decode = (S == 1 and the
// cache already holds the earlier positions).
int forward(fp_handle* h, const int32_t* tok, int S, bool decode) {
  const fp_arch& a = h->a;
  const int B = h->B, M = B * S, d = a.hidden;
  cudaStream_t s = h->stream;
  h->launches = 0;
  // kernels of one forward overlap their start-up with the previous kernel's tail
  struct PdlScope {
    PdlScope() { g_pdl = true; }
    ~PdlScope() { g_pdl = false; }
  } pdl_scope;
  h->tr.start();
  // the embedding and the first block's pre-attention RMSNorm in one kernel
  LTRY(launch_embed_rmsnorm(tok, M, h->embed, a.vocab, d, h->h, h->L[0].attn_norm, a.rms_eps, h->y, h->err, s),
       FP_K_EMBED);
  h->tr.boundary();
  for (int l = 0; l < a.n_layers; ++l) {
    Layer& Ly = h->L[l];
    const fp_kv_view kv = h->kv(l);
    if (l > 0) LTRY(launch_rmsnorm(h->h, M, d, 1, 0, Ly.attn_norm, a.rms_eps, h->y, s), FP_K_RMSNORM);
    const Mat& Q = Ly.mat[FP_M_QKV];
    LTRY(block_linear(h, FP_EPI_STORE, h->y, M, Q, nullptr, h->qkv), FP_K_LIN_QKV);
    LTRY(launch_rope_kv(h->qkv, B, S, h->n_qkv, a.n_heads, kv, h->pos, h->rope_cs, h->err, s), FP_K_ROPE_KV);
    if (decode) {
      cudaError_t e2 = cudaSuccess;
      cudaError_t e = launch_attention_decode(h->qkv, h->n_qkv, B, a.n_heads, kv, h->pos, 1, h->T, h->att,
                                              h->attn_ws, h->err, s, &e2);
      if (e != cudaSuccess) return h->cuda_fail(e, "attention decode");
      // the split kernel and the combine kernel (when there is one) are timed together
      h->launches += attention_decode_launches(B, a.n_kv_heads, a.head_dim, h->kvq, h->T);
      h->tr.after(FP_K_ATTN);
    } else {
      LTRY(launch_attention_prefill(h->qkv, h->n_qkv, B, S, a.n_heads, kv, h->att, h->err, s), FP_K_ATTN);
    }
    const Mat& O = Ly.mat[FP_M_O];
    LTRY(block_linear(h, FP_EPI_RESID, h->att, M, O, h->h, h->h), FP_K_LIN_O);
    LTRY(launch_rmsnorm(h->h, M, d, 1, 0, Ly.ffn_norm, a.rms_eps, h->y, s), FP_K_RMSNORM);
    const Mat& GU = Ly.mat[FP_M_GU];
    LTRY(block_linear(h, FP_EPI_SWIGLU, h->y, M, GU, nullptr, h->act), FP_K_LIN_GU);
    const Mat& D = Ly.mat[FP_M_DOWN];
    LTRY(block_linear(h, FP_EPI_RESID, h->act, M, D, h->h, h->h), FP_K_LIN_DOWN);
    if (h->hidden) {
      cudaError_t e = cudaMemcpyAsync(h->hidden + (size_t)l * h->max_rows * d, h->h, (size_t)M * d * 2,
                                      cudaMemcpyDeviceToDevice, s);
      if (e != cudaSuccess) return h->cuda_fail(e, "hidden copy");
    }
    h->tr.boundary();
  }
  LTRY(launch_rmsnorm(h->h, B, d, S, S - 1, h->final_norm, a.rms_eps, h->ylast, s), FP_K_RMSNORM);
  LTRY(launch_linear(FP_W_BF16, FP_EPI_F32, h->ylast, B, a.vocab, d, h->lm_head, nullptr, nullptr, nullptr,
                     h->logits, h->lin_ws, h->lin_ws_bytes, s, h->err),
       FP_K_LM_HEAD);
  // the greedy token, and each sequence's position moves past this pass
  LTRY(launch_argmax(h->logits, B, a.vocab, h->tokens, s, h->pos, S), FP_K_ARGMAX);
  h->tr.boundary();
  h->last_rows = M;
  return FP_OK;
}

int check_err_flag(fp_handle* h) {
  int32_t v = 0;
  cudaError_t e = cudaMemcpyAsync(&v, h->err, 4, cudaMemcpyDeviceToHost, h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return h->cuda_fail(e, "sync");
  if (v) {
    cudaMemsetAsync(h->err, 0, 4, h->stream);
    if (v == 2) return h->fail(FP_ERR_DEVICE_ASSERT, "a bounded wait in a pipelined kernel expired; its output is invalid");
    if (v == 3)
      return h->fail(FP_ERR_DEVICE_ASSERT,
                     "an activation beyond the fp16 range (|x| > 65504) reached a kernel that computes in fp16 "
                     "(an int8/int4 decode linear or the int8-cache prefill attention)");
    return h->fail(FP_ERR_DEVICE_ASSERT, "a kernel met an out-of-range token id or page id and skipped it");
  }
  return FP_OK;
}

int prefill_dev(fp_handle* h, int S) {
  cudaError_t e = cudaMemsetAsync(h->pos, 0, (size_t)h->B * 4, h->stream);
  if (e != cudaSuccess) return h->cuda_fail(e, "reset positions");
  int st = forward(h, h->prompt, S, false);
  if (st) return st;
  h->prefill_launches = h->launches;
  h->length = S;
  h->prefilled = true;
  return FP_OK;
}

int decode_dev(fp_handle* h) {
  if (!h->decode_exec) {
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaStreamBeginCapture(h->stream, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess) return h->cuda_fail(e, "begin capture");
    int st = forward(h, h->tokens, 1, true);
    e = cudaStreamEndCapture(h->stream, &g);
    if (st) {
      if (g) cudaGraphDestroy(g);
      return st;
    }
    if (e != cudaSuccess) return h->cuda_fail(e, "end capture");
    e = cudaGraphInstantiate(&h->decode_exec, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) {
      h->decode_exec = nullptr;
      return h->cuda_fail(e, "instantiate");
    }
  }
  cudaError_t e = cudaGraphLaunch(h->decode_exec, h->stream);
  if (e != cudaSuccess) return h->cuda_fail(e, "graph launch");
  h->length += 1;
  return FP_OK;
}

int upload_tokens(fp_handle* h, int32_t* dst, const int32_t* src, size_t n) {
  for (size_t i = 0; i < n; ++i)
    if (src[i] < 0 || src[i] >= h->a.vocab) return h->fail(FP_ERR_INVALID_ARG, "token id outside [0, vocab)");
  cudaError_t e = cudaMemcpyAsync(dst, src, n * 4, cudaMemcpyHostToDevice, h->stream);
  if (e != cudaSuccess) return h->cuda_fail(e, "upload tokens");
  return FP_OK;
}

int read_tokens(fp_handle* h, int32_t* out) {
  cudaError_t e = cudaMemcpyAsync(out, h->tokens, (size_t)h->B * 4, cudaMemcpyDeviceToHost, h->stream);
  if (e != cudaSuccess) return h->cuda_fail(e, "read tokens");
  return check_err_flag(h);
}

// Seeded weights: each tensor is its own SplitMix64 stream, (layer + 1) * 16 + tensor.
int init_weights(fp_handle* h, uint16_t* staging) {
  const fp_arch& a = h->a;
  cudaStream_t s = h->stream;
  const long long d = a.hidden, V = a.vocab;
  std::vector<uint16_t> one((size_t)d, 0x3F80);  // 1.0 in bf16
  cudaError_t e;
  e = launch_init_weights(h->embed, V * d, h->seed, 0 * 16 + FP_T_EMBED, 0, s);
  if (e == cudaSuccess) e = launch_init_weights(h->lm_head, V * d, h->seed, 0 * 16 + FP_T_LM_HEAD, 0, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(h->final_norm, one.data(), d * 2, cudaMemcpyHostToDevice, s);
  for (int l = 0; l < a.n_layers && e == cudaSuccess; ++l) {
    Layer& Ly = h->L[l];
    const long long base = (long long)(l + 1) * 16;
    e = cudaMemcpyAsync(Ly.attn_norm, one.data(), d * 2, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(Ly.ffn_norm, one.data(), d * 2, cudaMemcpyHostToDevice, s);
    // fused matrices: [Wq; Wk; Wv], Wo, [Wgate; Wup], Wdown
    const int parts[4][3] = {{FP_T_WQ, FP_T_WK, FP_T_WV}, {FP_T_WO, -1, -1}, {FP_T_WGATE, FP_T_WUP, -1},
                             {FP_T_WDOWN, -1, -1}};
    const long long rows[4][3] = {{h->q_dim, a.n_kv_heads * (long long)a.head_dim, a.n_kv_heads * (long long)a.head_dim},
                                  {d, 0, 0}, {a.ffn, a.ffn, 0}, {d, 0, 0}};
    for (int m = 0; m < 4 && e == cudaSuccess; ++m) {
      Mat& M = Ly.mat[m];
      long long r0 = 0;
      for (int p = 0; p < 3 && parts[m][p] >= 0 && e == cudaSuccess; ++p) {
        e = launch_init_weights(staging + r0 * M.K, rows[m][p] * M.K, h->seed, base + parts[m][p], 0, s);
        r0 += rows[m][p];
      }
      if (e == cudaSuccess) e = launch_quantize(h->wq, staging, M.N, M.K, M.codes, M.scales, M.zeros, s, M.perm);
      // the staging buffer is reused by the next matrix: keep the order
      if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    }
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return h->cuda_fail(e, "seeded weights");
  return FP_OK;
}

}  // namespace

// ====================================================================== C ABI
extern "C" {

const char* fp_strerror(int code) {
  switch (code) {
    case FP_OK: return "ok";
    case FP_ERR_INVALID_ARG: return "invalid argument";
    case FP_ERR_UNSUPPORTED: return "unsupported shape or mode";
    case FP_ERR_OOM: return "device allocation failed";
    case FP_ERR_CUDA: return "CUDA error";
    case FP_ERR_CAPACITY: return "KV cache capacity exceeded";
    case FP_ERR_DEVICE_ASSERT: return "device-side index check failed";
    case FP_ERR_STATE: return "call out of order";
    default: return "unknown status";
  }
}

const char* fp_last_error(const fp_handle* h) { return h ? h->msg.c_str() : g_create_error.c_str(); }

static int create_fail(fp_handle* h, int code, const std::string& m) {
  g_create_error = m;
  if (h) fp_destroy(h);
  return code;
}

int fp_create(const fp_arch* arch, int wquant, int kvquant, int batch, int max_context, int page_size,
              unsigned long long seed, unsigned flags, const fp_allocator* alloc, void* stream, fp_handle** out) {
  if (!out) return create_fail(nullptr, FP_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (!arch) return create_fail(nullptr, FP_ERR_INVALID_ARG, "arch is NULL");
  const fp_arch& a = *arch;
  if (a.n_layers < 1 || a.hidden <= 0 || a.n_heads <= 0 || a.n_kv_heads <= 0 || a.head_dim <= 0 || a.ffn <= 0 ||
      a.vocab <= 0 || !(a.rms_eps >= 0.f) || !(a.rope_base > 0.f))
    return create_fail(nullptr, FP_ERR_INVALID_ARG, "non-positive shape field or bad eps / rope base");
  if (a.n_heads % a.n_kv_heads != 0) return create_fail(nullptr, FP_ERR_INVALID_ARG, "n_heads % n_kv_heads != 0");
  if (wquant < FP_W_BF16 || wquant > FP_W_GPTQ4) return create_fail(nullptr, FP_ERR_INVALID_ARG, "wquant");
  if (kvquant != FP_KV_BF16 && kvquant != FP_KV_INT8) return create_fail(nullptr, FP_ERR_INVALID_ARG, "kvquant");
  if (batch < 1 || max_context < 1) return create_fail(nullptr, FP_ERR_INVALID_ARG, "batch and max_context >= 1");
  if (alloc && (!alloc->alloc || !alloc->free)) return create_fail(nullptr, FP_ERR_INVALID_ARG, "allocator fields");
  if (flags & ~(FP_FLAG_KEEP_HIDDEN | FP_FLAG_NO_INIT)) return create_fail(nullptr, FP_ERR_INVALID_ARG, "flags");
  if (a.n_layers > FP_MAX_LAYERS) return create_fail(nullptr, FP_ERR_UNSUPPORTED, "n_layers > FP_MAX_LAYERS");
  if (page_size != 16) return create_fail(nullptr, FP_ERR_UNSUPPORTED, "page_size must be 16");
  std::string why;
  if (bad_shape(arch, wquant, why)) return create_fail(nullptr, FP_ERR_UNSUPPORTED, why);
  if ((long long)batch * max_context > (1LL << 30))
    return create_fail(nullptr, FP_ERR_UNSUPPORTED, "batch * max_context above 2^30 rows");

  // ---- device from here on
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaFree(nullptr);
  if (e != cudaSuccess) return create_fail(nullptr, FP_ERR_CUDA, std::string("no usable CUDA device: ") + cudaGetErrorString(e));

  fp_handle* h = new fp_handle();
  h->a = a;
  h->wq = wquant;
  h->kvq = kvquant;
  h->B = batch;
  h->T = max_context;
  h->P = page_size;
  h->pps = (max_context + page_size - 1) / page_size;
  h->n_pages = batch * h->pps;
  h->seed = seed;
  h->flags = flags;
  h->max_rows = batch * max_context;
  h->q_dim = a.n_heads * a.head_dim;
  h->n_qkv = h->q_dim + 2 * a.n_kv_heads * a.head_dim;
  if (alloc) {
    h->alloc = *alloc;
    h->has_alloc = true;
  }
  if (stream) {
    h->stream = (cudaStream_t)stream;
  } else {
    e = cudaStreamCreateWithFlags(&h->stream, cudaStreamNonBlocking);
    if (e != cudaSuccess) return create_fail(h, FP_ERR_CUDA, "stream create");
    h->own_stream = true;
  }
  h->tr.s = h->stream;

  carve(h, nullptr);
  size_t free0 = 0, free1 = 0, total = 0;
  cudaMemGetInfo(&free0, &total);
  h->arena = h->dev_alloc(h->arena_bytes);
  if (!h->arena) {
    char buf[160];
    snprintf(buf, sizeof buf, "arena of %zu bytes could not be allocated", h->arena_bytes);
    return create_fail(h, FP_ERR_OOM, buf);
  }
  cudaMemGetInfo(&free1, &total);
  h->memgetinfo_bytes = free0 > free1 ? free0 - free1 : 0;
  h->free_before = free0;
  carve(h, (char*)h->arena);

  e = cudaMemsetAsync(h->arena, 0, h->arena_bytes, h->stream);
  if (e != cudaSuccess) return create_fail(h, FP_ERR_CUDA, "arena clear");
  std::vector<int32_t> pt((size_t)batch * h->pps);
  for (int b = 0; b < batch; ++b)
    for (int p = 0; p < h->pps; ++p) pt[(size_t)b * h->pps + p] = p * batch + b;
  e = cudaMemcpyAsync(h->page_table, pt.data(), pt.size() * 4, cudaMemcpyHostToDevice, h->stream);
  if (e != cudaSuccess) return create_fail(h, FP_ERR_CUDA, "page table upload");
  int st = fp_op_rope_table(h->pps * h->P, a.head_dim, a.rope_base, h->rope_cs, h->stream);
  if (st) return create_fail(h, st, "rope table");
  if (wquant == FP_W_GPTQ4) {
    // every matrix's act order, drawn from the seed on the host, and its inverse
    std::vector<int32_t> perm;
    for (int l = 0; l < a.n_layers && e == cudaSuccess; ++l)
      for (int m = 0; m < 4 && e == cudaSuccess; ++m) {
        const Mat& M = h->L[l].mat[m];
        perm.resize((size_t)M.K);
        act_order(seed, l, m, M.K, perm.data());
        e = cudaMemcpyAsync(M.perm, perm.data(), (size_t)M.K * 4, cudaMemcpyHostToDevice, h->stream);
        if (e == cudaSuccess) e = launch_invert_perm(M.perm, M.K, M.inv, nullptr, h->stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);  // the host buffer is reused
      }
    if (e != cudaSuccess) return create_fail(h, FP_ERR_CUDA, "act orders");
  }

  if (!(flags & FP_FLAG_NO_INIT)) {
    size_t stage = 0;
    for (int m = 0; m < 4; ++m) stage = std::max(stage, (size_t)h->L[0].mat[m].N * h->L[0].mat[m].K * 2);
    uint16_t* staging = (uint16_t*)h->dev_alloc(stage);
    if (!staging) return create_fail(h, FP_ERR_OOM, "weight staging buffer");
    st = init_weights(h, staging);
    cudaStreamSynchronize(h->stream);
    h->dev_free(staging);
    if (st) return create_fail(h, st, h->msg);
  }
  e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return create_fail(h, FP_ERR_CUDA, std::string("create: ") + cudaGetErrorString(e));
  *out = h;
  return FP_OK;
}

void fp_destroy(fp_handle* h) {
  if (!h) return;
  if (h->stream) cudaStreamSynchronize(h->stream);
  h->tr.clear();
  if (h->decode_exec) cudaGraphExecDestroy(h->decode_exec);
  h->dev_free(h->arena);
  if (h->own_stream && h->stream) cudaStreamDestroy(h->stream);
  delete h;
}

int fp_get_plan(const fp_handle* h, fp_plan* out) {
  if (!h || !out) return FP_ERR_INVALID_ARG;
  out->weight_bytes = h->weight_bytes;
  out->kv_bytes = h->kv_bytes;
  out->act_bytes = h->act_bytes;
  out->workspace_bytes = h->ws_bytes;
  out->total_bytes = h->arena_bytes;
  out->pages_per_seq = h->pps;
  out->max_rows = h->max_rows;
  return FP_OK;
}

int fp_set_weight(fp_handle* h, int layer, int tensor, const uint16_t* host_bf16, size_t n_elems) {
  if (!h) return FP_ERR_INVALID_ARG;
  if (!host_bf16) return h->fail(FP_ERR_INVALID_ARG, "host_bf16 is NULL");
  const fp_arch& a = h->a;
  const long long d = a.hidden, f = a.ffn, V = a.vocab, kvd = (long long)a.n_kv_heads * a.head_dim;
  cudaStream_t s = h->stream;
  cudaError_t e;
  if (layer == -1) {
    uint16_t* dst = nullptr;
    long long n = 0;
    if (tensor == FP_T_EMBED) { dst = h->embed; n = V * d; }
    else if (tensor == FP_T_FINAL_NORM) { dst = h->final_norm; n = d; }
    else if (tensor == FP_T_LM_HEAD) { dst = h->lm_head; n = V * d; }
    else return h->fail(FP_ERR_INVALID_ARG, "global tensor id");
    if ((long long)n_elems != n) return h->fail(FP_ERR_INVALID_ARG, "n_elems does not match the tensor");
    e = cudaMemcpyAsync(dst, host_bf16, n * 2, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    return e == cudaSuccess ? FP_OK : h->cuda_fail(e, "set weight");
  }
  if (layer < 0 || layer >= a.n_layers) return h->fail(FP_ERR_INVALID_ARG, "layer out of range");
  Layer& Ly = h->L[layer];
  if (tensor == FP_T_ATTN_NORM || tensor == FP_T_FFN_NORM) {
    if ((long long)n_elems != d) return h->fail(FP_ERR_INVALID_ARG, "n_elems does not match the tensor");
    e = cudaMemcpyAsync(tensor == FP_T_ATTN_NORM ? Ly.attn_norm : Ly.ffn_norm, host_bf16, d * 2,
                        cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    return e == cudaSuccess ? FP_OK : h->cuda_fail(e, "set weight");
  }
  int m;
  long long r0, rows;
  switch (tensor) {
    case FP_T_WQ: m = FP_M_QKV; r0 = 0; rows = h->q_dim; break;
    case FP_T_WK: m = FP_M_QKV; r0 = h->q_dim; rows = kvd; break;
    case FP_T_WV: m = FP_M_QKV; r0 = h->q_dim + kvd; rows = kvd; break;
    case FP_T_WO: m = FP_M_O; r0 = 0; rows = d; break;
    case FP_T_WGATE: m = FP_M_GU; r0 = 0; rows = f; break;
    case FP_T_WUP: m = FP_M_GU; r0 = f; rows = f; break;
    case FP_T_WDOWN: m = FP_M_DOWN; r0 = 0; rows = d; break;
    default: return h->fail(FP_ERR_INVALID_ARG, "layer tensor id");
  }
  Mat& M = Ly.mat[m];
  if ((long long)n_elems != rows * M.K) return h->fail(FP_ERR_INVALID_ARG, "n_elems does not match the tensor");
  uint16_t* staging = (uint16_t*)h->dev_alloc((size_t)rows * M.K * 2);
  if (!staging) return h->fail(FP_ERR_OOM, "staging buffer for set_weight");
  const int wq = h->wq;
  char* codes = (char*)M.codes + codes_bytes(wq, r0, M.K);
  uint16_t* sc = M.scales ? (uint16_t*)((char*)M.scales + scale_bytes(wq, r0, M.K)) : nullptr;
  uint16_t* zr = M.zeros ? (uint16_t*)((char*)M.zeros + zero_bytes(wq, r0, M.K)) : nullptr;
  e = cudaMemcpyAsync(staging, host_bf16, (size_t)rows * M.K * 2, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = launch_quantize(wq, staging, (int)rows, M.K, codes, sc, zr, s, M.perm);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  h->dev_free(staging);
  return e == cudaSuccess ? FP_OK : h->cuda_fail(e, "set weight");
}

int fp_set_page_table(fp_handle* h, const int32_t* host_table) {
  if (!h) return FP_ERR_INVALID_ARG;
  if (!host_table) return h->fail(FP_ERR_INVALID_ARG, "host_table is NULL");
  const size_t n = (size_t)h->B * h->pps;
  std::vector<char> used((size_t)h->n_pages, 0);
  for (size_t i = 0; i < n; ++i) {
    const int p = host_table[i];
    if (p < 0 || p >= h->n_pages) return h->fail(FP_ERR_INVALID_ARG, "page id outside the pool");
    if (used[p]) return h->fail(FP_ERR_INVALID_ARG, "page id used twice");
    used[p] = 1;
  }
  cudaError_t e = cudaMemcpyAsync(h->page_table, host_table, n * 4, cudaMemcpyHostToDevice, h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  return e == cudaSuccess ? FP_OK : h->cuda_fail(e, "page table");
}

int fp_load_prompt(fp_handle* h, const int32_t* host_tokens, int prompt_len) {
  if (!h) return FP_ERR_INVALID_ARG;
  if (prompt_len < 1) return h->fail(FP_ERR_INVALID_ARG, "prompt_len < 1");
  if (prompt_len > h->T) return h->fail(FP_ERR_CAPACITY, "prompt longer than max_context");
  const size_t n = (size_t)h->B * prompt_len;
  std::vector<int32_t> gen;
  if (!host_tokens) {
    // SplitMix64 stream 2^20 of the seed, multiply-shift onto [0, vocab)
    gen.resize(n);
    const uint64_t key = stream_key(h->seed, 1ull << 20);
    for (size_t i = 0; i < n; ++i) {
      const uint64_t u = mix64(key + (uint64_t)(i + 1) * kGamma);
      gen[i] = (int32_t)(((u >> 32) * (uint64_t)h->a.vocab) >> 32);
    }
    host_tokens = gen.data();
  }
  int st = upload_tokens(h, h->prompt, host_tokens, n);
  if (st) return st;
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return h->cuda_fail(e, "load prompt");
  h->prompt_len = prompt_len;
  return FP_OK;
}

int fp_prefill(fp_handle* h, const int32_t* host_tokens, int prompt_len, int32_t* host_next) {
  if (!h) return FP_ERR_INVALID_ARG;
  if (prompt_len < 1) return h->fail(FP_ERR_INVALID_ARG, "prompt_len < 1");
  if (prompt_len > h->T) return h->fail(FP_ERR_CAPACITY, "prompt longer than max_context");
  if (host_tokens) {
    int st = upload_tokens(h, h->prompt, host_tokens, (size_t)h->B * prompt_len);
    if (st) return st;
    h->prompt_len = prompt_len;
  } else if (prompt_len != h->prompt_len) {
    return h->fail(FP_ERR_STATE, "no resident prompt of that length (fp_load_prompt)");
  }
  int st = prefill_dev(h, prompt_len);
  if (st) return st;
  return host_next ? read_tokens(h, host_next) : FP_OK;
}

int fp_decode_steps(fp_handle* h, int n) {
  if (!h) return FP_ERR_INVALID_ARG;
  if (n < 0) return h->fail(FP_ERR_INVALID_ARG, "n < 0");
  if (!h->prefilled) return h->fail(FP_ERR_STATE, "decode before prefill");
  if (h->length + n > h->T) return h->fail(FP_ERR_CAPACITY, "KV cache is full");
  for (int i = 0; i < n; ++i) {
    int st = decode_dev(h);
    if (st) return st;
  }
  return FP_OK;
}

int fp_decode_step(fp_handle* h, const int32_t* host_in, int32_t* host_out) {
  if (!h) return FP_ERR_INVALID_ARG;
  if (!h->prefilled) return h->fail(FP_ERR_STATE, "decode before prefill");
  if (h->length + 1 > h->T) return h->fail(FP_ERR_CAPACITY, "KV cache is full");
  if (host_in) {
    int st = upload_tokens(h, h->tokens, host_in, (size_t)h->B);
    if (st) return st;
  }
  int st = decode_dev(h);
  if (st) return st;
  return host_out ? read_tokens(h, host_out) : FP_OK;
}

long long fp_get_tensor(fp_handle* h, int what, int layer, int mat, void* host_dst, size_t bytes) {
  return fp_get_tensor_at(h, what, layer, mat, 0, host_dst, bytes);
}

long long fp_get_tensor_at(fp_handle* h, int what, int layer, int mat, size_t offset, void* host_dst, size_t bytes) {
  if (!h) return FP_ERR_INVALID_ARG;
  const void* src = nullptr;
  size_t n = 0;
  const bool per_layer = what <= FP_G_HIDDEN || what == FP_G_W_PERM;
  if (per_layer && (layer < 0 || layer >= h->a.n_layers)) return h->fail(FP_ERR_INVALID_ARG, "layer out of range");
  const size_t pool = (size_t)h->n_pages * h->a.n_kv_heads * h->P * h->a.head_dim * (h->kvq == FP_KV_BF16 ? 2 : 1);
  const size_t spool = (size_t)h->n_pages * h->a.n_kv_heads * h->P * 4;
  switch (what) {
    case FP_G_W_CODES:
    case FP_G_W_SCALES:
    case FP_G_W_ZEROS: {
      if (mat < 0 || mat > 3) return h->fail(FP_ERR_INVALID_ARG, "mat out of range");
      const Mat& M = h->L[layer].mat[mat];
      if (what == FP_G_W_CODES) { src = M.codes; n = codes_bytes(h->wq, M.N, M.K); }
      else if (what == FP_G_W_SCALES) { src = M.scales; n = scale_bytes(h->wq, M.N, M.K); }
      else { src = M.zeros; n = zero_bytes(h->wq, M.N, M.K); }
      break;
    }
    case FP_G_W_PERM: {
      if (mat < 0 || mat > 3) return h->fail(FP_ERR_INVALID_ARG, "mat out of range");
      const Mat& M = h->L[layer].mat[mat];
      src = M.perm;
      n = perm_bytes(h->wq, M.K);
      break;
    }
    case FP_G_K_POOL: src = h->L[layer].kpool; n = pool; break;
    case FP_G_V_POOL: src = h->L[layer].vpool; n = pool; break;
    case FP_G_K_SCALES: src = h->L[layer].kscale; n = src ? spool : 0; break;
    case FP_G_V_SCALES: src = h->L[layer].vscale; n = src ? spool : 0; break;
    case FP_G_HIDDEN:
      if (!h->hidden) return h->fail(FP_ERR_STATE, "created without FP_FLAG_KEEP_HIDDEN");
      src = h->hidden + (size_t)layer * h->max_rows * h->a.hidden;
      n = (size_t)h->last_rows * h->a.hidden * 2;
      break;
    case FP_G_LOGITS: src = h->logits; n = (size_t)h->B * h->a.vocab * 4; break;
    case FP_G_TOKENS: src = h->tokens; n = (size_t)h->B * 4; break;
    case FP_G_PAGE_TABLE: src = h->page_table; n = (size_t)h->B * h->pps * 4; break;
    case FP_G_LENGTH: src = h->pos; n = (size_t)h->B * 4; break;
    default: return h->fail(FP_ERR_INVALID_ARG, "unknown tensor");
  }
  if (offset > n) return h->fail(FP_ERR_INVALID_ARG, "offset past the end of the tensor");
  if (!host_dst) return (long long)(n - offset);
  n = std::min(n - offset, bytes);  // a smaller buffer receives the leading bytes from offset on
  if (n == 0) return 0;
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e == cudaSuccess) e = cudaMemcpy(host_dst, (const char*)src + offset, n, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return h->cuda_fail(e, "get tensor");
  return (long long)n;
}

// Algorithmic bytes: block matrices (codes + scales/zeros), K/V of every
// cached position, and the bf16 LM head; the closed forms of the byte model.
static unsigned long long block_matrix_bytes(const fp_handle* h) {
  unsigned long long t = 0;
  for (int m = 0; m < 4; ++m) {
    const Mat& M = h->L[0].mat[m];
    t += codes_bytes(h->wq, M.N, M.K) + scale_bytes(h->wq, M.N, M.K) + zero_bytes(h->wq, M.N, M.K) +
         perm_bytes(h->wq, M.K);
  }
  return t;
}
static unsigned long long kv_token_bytes(const fp_handle* h) {
  const unsigned long long r = (unsigned long long)h->a.n_kv_heads * h->a.head_dim;
  return h->kvq == FP_KV_BF16 ? 2 * r * 2 : 2 * r + 2ull * h->a.n_kv_heads * 4;
}

int fp_profile(fp_handle* h, int prompt_len, int n_decode, int warmup, int iters, const int32_t* host_prompt,
               fp_profile_result* out) {
  if (!h) return FP_ERR_INVALID_ARG;
  if (!out) return h->fail(FP_ERR_INVALID_ARG, "out is NULL");
  if (prompt_len < 1 || n_decode < 0 || warmup < 0 || iters < 1)
    return h->fail(FP_ERR_INVALID_ARG, "prompt_len >= 1, n_decode >= 0, warmup >= 0, iters >= 1");
  if (prompt_len + n_decode > h->T) return h->fail(FP_ERR_CAPACITY, "prompt_len + n_decode > max_context");
  memset(out, 0, sizeof *out);
  const int B = h->B;
  int st = fp_load_prompt(h, host_prompt, prompt_len);
  if (st) return st;
  // make sure the decode graph exists before anything is timed
  if (!h->decode_exec && n_decode > 0 && prompt_len + 1 <= h->T) {
    if ((st = prefill_dev(h, prompt_len)) || (st = decode_dev(h))) return st;
  }
  for (int w = 0; w < warmup; ++w) {
    if ((st = prefill_dev(h, prompt_len))) return st;
    for (int j = 0; j < n_decode; ++j)
      if ((st = decode_dev(h))) return st;
  }
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return h->cuda_fail(e, "warmup");
  std::vector<cudaEvent_t> ev((size_t)iters * (n_decode + 2));
  for (auto& x : ev) cudaEventCreate(&x);
  double ttft = 0, dec = 0, req = 0;
  std::vector<double> steps;
  for (int it = 0; it < iters && !st; ++it) {
    cudaEvent_t* E = &ev[(size_t)it * (n_decode + 2)];
    cudaEventRecord(E[0], h->stream);
    st = prefill_dev(h, prompt_len);
    cudaEventRecord(E[1], h->stream);
    for (int j = 0; j < n_decode && !st; ++j) {
      st = decode_dev(h);
      cudaEventRecord(E[2 + j], h->stream);
    }
  }
  e = cudaStreamSynchronize(h->stream);
  if (!st && e != cudaSuccess) st = h->cuda_fail(e, "timed passes");
  if (!st) {
    for (int it = 0; it < iters; ++it) {
      cudaEvent_t* E = &ev[(size_t)it * (n_decode + 2)];
      float ms = 0;
      cudaEventElapsedTime(&ms, E[0], E[1]);
      ttft += ms;
      cudaEventElapsedTime(&ms, E[0], E[1 + n_decode]);
      req += ms;
      for (int j = 0; j < n_decode; ++j) {
        cudaEventElapsedTime(&ms, E[1 + j], E[2 + j]);
        steps.push_back(ms);
        dec += ms;
      }
    }
  }
  for (auto& x : ev) cudaEventDestroy(x);
  if (st) return st;
  if ((st = check_err_flag(h))) return st;
  const fp_arch& a = h->a;
  out->ttft_ms = ttft / iters;
  out->request_ms = req / iters;
  out->n_layers = a.n_layers;
  out->prompt_len = prompt_len;
  out->n_decode = n_decode;
  out->iters = iters;
  if (n_decode > 0) {
    out->tpot_ms = dec / steps.size();
    std::vector<double> srt = steps;
    std::sort(srt.begin(), srt.end());
    out->tpot_ms_p50 = srt[srt.size() / 2];
    out->decode_tokens_per_s = (double)B * steps.size() / (dec * 1e-3);
  }
  // algorithmic prefill FLOPs: linear layers, causal attention, LM head on the last rows
  double params = 0;
  for (int m = 0; m < 4; ++m) params += (double)h->L[0].mat[m].N * h->L[0].mat[m].K;
  out->prefill_flops = 2.0 * B * prompt_len * params * a.n_layers +
                       2.0 * B * a.n_heads * (double)prompt_len * prompt_len * a.head_dim * a.n_layers +
                       2.0 * B * (double)a.vocab * a.hidden;
  out->prefill_tflops = out->ttft_ms > 0 ? out->prefill_flops / (out->ttft_ms * 1e-3) / 1e12 : 0;
  const double mean_ctx = prompt_len + (n_decode + 1) / 2.0;
  out->decode_bytes_per_step =
      (unsigned long long)(a.n_layers * (block_matrix_bytes(h) + B * mean_ctx * kv_token_bytes(h)) +
                           2.0 * a.vocab * a.hidden);
  out->peak_hbm_bytes = h->arena_bytes;
  out->weight_bytes = h->weight_bytes;
  out->kv_bytes = h->kv_bytes;
  out->act_bytes = h->act_bytes;
  out->workspace_bytes = h->ws_bytes;
  out->memgetinfo_bytes = h->memgetinfo_bytes;

  // ---- instrumented eager decode steps: events between kernels
  const int ksteps = std::min(n_decode, 8);
  if (ksteps > 0) {
    if ((st = prefill_dev(h, prompt_len))) return st;
    cudaStreamSynchronize(h->stream);
    double blk[FP_MAX_LAYERS] = {0}, other = 0, kms[FP_K_COUNT] = {0};
    int kl[FP_K_COUNT] = {0};
    for (int j = 0; j < ksteps && !st; ++j) {
      h->tr.on = true;
      st = forward(h, h->tokens, 1, true);
      h->tr.on = false;
      h->length += 1;
      if (st) break;
      e = cudaStreamSynchronize(h->stream);
      if (e != cudaSuccess) { st = h->cuda_fail(e, "instrumented step"); break; }
      Tracer& T = h->tr;
      for (size_t i = 1; i < T.ev.size(); ++i) {
        float ms = 0;
        cudaEventElapsedTime(&ms, T.ev[i - 1], T.ev[i]);
        kms[T.cls[i]] += ms;
        if (j == 0) kl[T.cls[i]] += 1;
      }
      // marks: after embed, after each block, after the head
      float ms = 0;
      cudaEventElapsedTime(&ms, T.ev[0], T.ev[T.mark[0]]);
      other += ms;
      for (int l = 0; l < a.n_layers; ++l) {
        cudaEventElapsedTime(&ms, T.ev[T.mark[l]], T.ev[T.mark[l + 1]]);
        blk[l] += ms;
      }
      cudaEventElapsedTime(&ms, T.ev[T.mark[a.n_layers]], T.ev[T.mark[a.n_layers + 1]]);
      other += ms;
      T.clear();
    }
    h->tr.clear();
    if (st) return st;
    const double ctx = prompt_len + (ksteps + 1) / 2.0;
    for (int l = 0; l < a.n_layers; ++l) {
      out->block_ms[l] = blk[l] / ksteps;
      out->block_bytes[l] = (unsigned long long)(block_matrix_bytes(h) + B * ctx * kv_token_bytes(h));
    }
    out->other_ms = other / ksteps;
    out->decode_launches = h->launches;
    out->prefill_launches = h->prefill_launches;
    for (int k = 0; k < FP_K_COUNT; ++k) {
      out->kernel_ms[k] = kms[k] / ksteps;
      out->kernel_launches[k] = kl[k];
    }
  }
  // observed: the device memory the deployment holds now, after its passes
  // (arena, decode graph, loaded kernels), as a monitor of the GPU sees it
  {
    size_t free_now = 0, total = 0;
    if (cudaMemGetInfo(&free_now, &total) == cudaSuccess && h->free_before > free_now)
      out->observed_hbm_bytes = h->free_before - free_now;
  }
  return check_err_flag(h);
}

}  // extern "C"
