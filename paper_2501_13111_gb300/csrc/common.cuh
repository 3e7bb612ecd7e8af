// Shared device helpers of the fingerprint kernels (bf16 bit handling,
// warp reductions, vector loads).  Every kernel of the library is written
// for sm_103a only.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#define FP_DEV __device__ __forceinline__
#define FP_HD __host__ __device__ __forceinline__

namespace fpk {

// bf16 stored as uint16 bit patterns across the whole library.
FP_HD float bf2f(uint16_t b) {
#ifdef __CUDA_ARCH__
  return __uint_as_float(((uint32_t)b) << 16);
#else
  uint32_t u = ((uint32_t)b) << 16;
  float f;
  __builtin_memcpy(&f, &u, 4);
  return f;
#endif
}

// fp32 -> bf16, round to nearest even (finite inputs).
FP_DEV uint16_t f2bf(float f) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

// Smallest bf16 >= x for x >= 0 (bf16 rounding toward +inf).
FP_DEV uint16_t f2bf_ceil(float x) {
  uint32_t b = __float_as_uint(x);
  uint32_t hi = b >> 16;
  return (uint16_t)(hi + ((b & 0xFFFFu) != 0u ? 1u : 0u));
}

// Two bf16 packed in a uint32 (low half = first element).
FP_DEV float2 bf2x2f(uint32_t v) {
  return make_float2(__uint_as_float(v << 16), __uint_as_float(v & 0xFFFF0000u));
}

FP_DEV uint32_t pack_bf2(float a, float b) {
  return (uint32_t)f2bf(a) | ((uint32_t)f2bf(b) << 16);
}

FP_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

FP_DEV float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// 16-byte streaming load that does not allocate in L1 (weights are read once).
FP_DEV uint4 ld_stream16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

FP_DEV uint4 ld_nc16(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }

FP_DEV float silu(float x) { return x / (1.0f + __expf(-x)); }

// Programmatic dependent launch: a kernel launched with programmatic stream
// serialisation may start while the previous kernel in the stream is still
// running.  pdl_trigger() lets the next kernel be scheduled; pdl_wait()
// blocks until the previous kernel has completed and its writes are visible
// (a no-op when the kernel was launched without the attribute).  Every
// kernel of the forward pass waits before it touches activations, caches or
// workspaces; only reads of the constant weights may come before the wait.
FP_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
FP_DEV void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Set by the runtime while it enqueues a forward pass: launches then carry
// the programmatic-serialisation attribute.
extern thread_local bool g_pdl;

template <typename... KArgs, typename... Args>
inline cudaError_t launch(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                          Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = g_pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// Lifts a kernel's dynamic shared-memory limit to `bytes` once per device:
// function attributes belong to each device's context, so a process that
// drives several GPUs sets it on each.  `done` (one per call site) holds a
// bit per device ordinal below 64.
template <typename... KArgs>
inline cudaError_t smem_limit_once(void (*kern)(KArgs...), int bytes, std::atomic<unsigned long long>* done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = 1ull << (dev & 63);
  if (done->load(std::memory_order_acquire) & bit) return cudaSuccess;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done->fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

// SplitMix64 finaliser (Steele, Lea and Flood, OOPSLA 2014).  The generator's
// state advances by kGamma; output i of a stream keyed by K is
// mix64(K + (i + 1) * kGamma), so draws are counter-based.
static constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
FP_HD uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
FP_HD uint64_t stream_key(uint64_t seed, uint64_t stream) { return mix64(seed + (stream + 1) * kGamma); }

}  // namespace fpk

// Host-side helpers
#define FP_CUDA_TRY(expr)                         \
  do {                                            \
    cudaError_t e__ = (expr);                     \
    if (e__ != cudaSuccess) return e__;           \
  } while (0)

static inline int fp_ceil_div(long long a, long long b) { return (int)((a + b - 1) / b); }
