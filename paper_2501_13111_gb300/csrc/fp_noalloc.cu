// Decode attention for callers that cannot allocate device memory.
//
// fp_op_attention_decode needs a caller-provided workspace for the partial
// results of its context splits.  Some callers have no way to provide one: a
// host program whose device memory is entirely reserved up front by another
// framework's pool (so an extra cudaMalloc fails or breaks its accounting), a
// plugin that must not call into the allocator from its execution hook, or a
// latency-critical loop that cannot afford the implicit synchronisation a
// cudaMalloc / cudaFree may cause.  This file gives them the same kernels with
// the scratch held in a fixed-size array that lives in the library itself.
//
// The array is a file-scope __device__ variable: every GPU on which the
// library's module is loaded holds FP_NOALLOC_SCRATCH_BYTES for it until the
// process exits.  Host code cannot use the array's name as a device address
// (on the host it names a host-side stand-in), so the device address is looked
// up with cudaGetSymbolAddress, with the device current, and cached per device
// together with the id of the context it was looked up in.  A device reset
// (cudaDeviceReset) ends that context; the next call then runs in a new
// context, whose id differs, and looks the address up again instead of using
// one that belonged to the old context.
#include <cuda.h>

#include <mutex>

#include "common.cuh"
#include "kernels.cuh"

extern int fpk_check_kv(const fp_kv_view* kv);

static __device__ __align__(256) unsigned char g_decode_scratch[FP_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
struct ScratchAddr {
  void* ptr = nullptr;
  unsigned long long ctx_id = 0;
};
ScratchAddr g_scratch_addr[kMaxDevices];

// Id of the calling thread's current context (unique over the process's
// lifetime; cuCtxGetId), reached through the runtime's driver entry points so
// that the library needs no link-time dependency on libcuda.  0 if unknown.
unsigned long long current_context_id() {
  typedef CUresult (*GetCurrentFn)(CUcontext*);
  typedef CUresult (*GetIdFn)(CUcontext, unsigned long long*);
  static GetCurrentFn get_current = nullptr;
  static GetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPoint("cuCtxGetCurrent", &p, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = (GetCurrentFn)p;
    p = nullptr;
    if (cudaGetDriverEntryPoint("cuCtxGetId", &p, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = (GetIdFn)p;
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

// Device address of g_decode_scratch on the current device.  The first call
// on a device (and the first after its context was replaced) looks it up and
// caches it; a context whose id cannot be read is looked up on every call.
int scratch_on_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return FP_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return FP_ERR_UNSUPPORTED;
  const unsigned long long id = current_context_id();  // 0 before the runtime has made a context current
  std::lock_guard<std::mutex> lock(g_mu);
  ScratchAddr& a = g_scratch_addr[dev];
  if (!a.ptr || id == 0 || a.ctx_id != id) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_decode_scratch);  // with the device's primary context current
    if (e != cudaSuccess || !p) return FP_ERR_CUDA;
    a.ptr = p;
    a.ctx_id = id ? id : current_context_id();
  }
  *out = a.ptr;
  return FP_OK;
}

}  // namespace

extern "C" int fp_op_attention_decode_noalloc(const uint16_t* q, int q_stride, int B, int n_heads,
                                              const fp_kv_view* kv, const int32_t* len, int max_len,
                                              uint16_t* out, int32_t* err, void* stream) {
  int st = fpk_check_kv(kv);
  if (st) return st;
  if (!q || !len || !out || B < 0 || n_heads <= 0 || max_len <= 0) return FP_ERR_INVALID_ARG;
  if (n_heads % kv->n_kv_heads != 0) return FP_ERR_INVALID_ARG;
  const int G = n_heads / kv->n_kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8) return FP_ERR_UNSUPPORTED;
  if (q_stride < n_heads * kv->head_dim) return FP_ERR_INVALID_ARG;
  if (max_len > kv->pages_per_seq * kv->page_size) return FP_ERR_CAPACITY;
  if (B == 0) return FP_OK;
  // The same bound the allocating entry point asks its caller to provide.
  if (fpk::attention_decode_ws_bytes(B, n_heads, kv->head_dim, max_len) > (size_t)FP_NOALLOC_SCRATCH_BYTES)
    return FP_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  st = scratch_on_current_device(&scratch);
  if (st) return st;
  // Every partial the combine kernel reads is written by the same call, so the
  // scratch needs no clearing between calls.  Calls that overlap on the GPU
  // share the array and race on it.
  cudaError_t e = fpk::launch_attention_decode(q, q_stride, B, n_heads, *kv, len, 0, max_len, out, scratch, err,
                                               (cudaStream_t)stream);
  return e == cudaSuccess ? FP_OK : FP_ERR_CUDA;
}
