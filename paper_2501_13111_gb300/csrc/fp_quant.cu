// Seeded weight fill and weight-only quantisers (run at fp_create /
// fp_set_weight, off the timed path).
//
// Formats are the ones fp.h documents for the paper's INT8 / INT4 weight-only
// configurations (Sec. 3.2; table "Models and configurations").  Every
// rounding decision uses IEEE fp32 division (__fdiv_rn) and rintf (ties to
// even), so the codes are bit-identical to any other implementation of the
// same definition.
#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"

namespace fpk {

// Irwin-Hall(4) approximate normal, sigma 0.02: the four 16-bit lanes of a
// draw are summed, centred (mean 131070) and scaled by
// 0.02 / sqrt(4 (65536^2 - 1) / 12) in one fp64 multiplication, then rounded
// to fp32 and to bf16 (both to nearest even).
__global__ void init_weights_kernel(uint16_t* __restrict__ w, long long n, uint64_t key, long long start) {
  const double kScale = 0x1.1bc779ef9b324p-21;
  long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    uint64_t u = mix64(key + (uint64_t)(start + i + 1) * kGamma);
    long long s = (long long)(u & 0xFFFF) + (long long)((u >> 16) & 0xFFFF) + (long long)((u >> 32) & 0xFFFF) +
                  (long long)(u >> 48);
    double v = __dmul_rn((double)(s - 131070), kScale);
    w[i] = f2bf(__double2float_rn(v));
  }
}

cudaError_t launch_init_weights(uint16_t* w, long long n, unsigned long long seed, long long stream_id,
                                long long start, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  uint64_t key = stream_key((uint64_t)seed, (uint64_t)stream_id);
  int blocks = (int)((n + 255) / 256);
  if (blocks > 152 * 16) blocks = 152 * 16;
  return launch(init_weights_kernel, dim3(blocks), dim3(256), 0, s, w, n, key, start);
}

// ------------------------------------------------------------------ int8 rows
// One CTA per output row: s = bf16_ceil(fp32(amax / 127)),
// q = clamp(rint(fp32(w / s)), -127, 127); a zero row gives s = 0, q = 0.
__global__ void quantize_int8_kernel(const uint16_t* __restrict__ w, int K, int8_t* __restrict__ q,
                                     uint16_t* __restrict__ scales) {
  const long long row = blockIdx.x;
  const uint16_t* wr = w + row * K;
  float amax = 0.f;
  for (int k = threadIdx.x; k < K; k += blockDim.x) amax = fmaxf(amax, fabsf(bf2f(wr[k])));
  amax = warp_max(amax);
  __shared__ float red[32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = amax;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
    v = warp_max(v);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  amax = red[0];
  uint16_t sb = f2bf_ceil(__fdiv_rn(amax, 127.0f));
  float sc = bf2f(sb);
  if (threadIdx.x == 0) scales[row] = sb;
  int8_t* qr = q + row * K;
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    float r = sc > 0.f ? rintf(__fdiv_rn(bf2f(wr[k]), sc)) : 0.f;
    r = fminf(fmaxf(r, -127.f), 127.f);
    qr[k] = (int8_t)(int)r;
  }
}

// ------------------------------------------------------------------ int4 g128
// One warp per (row, 128-wide group); lane i holds elements 4i .. 4i+3.
// mn = min(0, min w), mx = max(0, max w), s = bf16_ceil(fp32(fp32(mx - mn) / 15)),
// z = clamp(rint(fp32(-mn / s)), 0, 15), q = clamp(rint(fp32(w / s)) + z, 0, 15).
// perm (GPTQ4, may be NULL): element j of the stored row is input channel
// perm[j], so group g holds channels perm[128 g .. 128 g + 127] (act order).
__global__ void quantize_int4_kernel(const uint16_t* __restrict__ w, int N, int K, uint8_t* __restrict__ q,
                                     uint16_t* __restrict__ scales, uint16_t* __restrict__ zeros,
                                     const int32_t* __restrict__ perm) {
  const int groups = K / 128;
  long long gid = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (gid >= (long long)N * groups) return;
  const int lane = threadIdx.x & 31;
  const long long row = gid / groups;
  const int g = (int)(gid % groups);
  float v[4];
  if (perm) {
    // an entry outside [0, K) reads as 0 (the act order must be a permutation)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int k = perm[g * 128 + lane * 4 + i];
      v[i] = (unsigned)k < (unsigned)K ? bf2f(w[row * K + k]) : 0.f;
    }
  } else {
    const uint2 raw = *reinterpret_cast<const uint2*>(w + row * K + g * 128 + lane * 4);
    v[0] = __uint_as_float(raw.x << 16);
    v[1] = __uint_as_float(raw.x & 0xFFFF0000u);
    v[2] = __uint_as_float(raw.y << 16);
    v[3] = __uint_as_float(raw.y & 0xFFFF0000u);
  }
  float mn = fminf(fminf(v[0], v[1]), fminf(v[2], v[3]));
  float mx = fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  mn = fminf(mn, 0.f);
  mx = fmaxf(mx, 0.f);
  float d = __fsub_rn(mx, mn);
  uint16_t sb = f2bf_ceil(__fdiv_rn(d, 15.0f));
  float sc = bf2f(sb);
  float z = 0.f;
  if (sc > 0.f) z = fminf(fmaxf(rintf(__fdiv_rn(-mn, sc)), 0.f), 15.f);
  uint32_t c[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float r = sc > 0.f ? __fadd_rn(rintf(__fdiv_rn(v[i], sc)), z) : 0.f;
    c[i] = (uint32_t)fminf(fmaxf(r, 0.f), 15.f);
  }
  // Word w of the group holds elements 8w .. 8w+7 (lanes 2w and 2w+1); nibble
  // i holds element (0,2,4,6,1,3,5,7)[i], i.e. element e sits in nibble
  // (e >> 1) + 4 (e & 1).
  const bool odd = lane & 1;
  const uint32_t part = odd ? ((c[0] << 8) | (c[2] << 12) | (c[1] << 24) | (c[3] << 28))
                            : (c[0] | (c[2] << 4) | (c[1] << 16) | (c[3] << 20));
  const uint32_t word = part | __shfl_xor_sync(0xffffffffu, part, 1);
  if (!odd) *reinterpret_cast<uint32_t*>(q + row * (K / 2) + g * 64 + (lane >> 1) * 4) = word;
  if (lane == 0) {
    scales[row * groups + g] = sb;
    zeros[row * groups + g] = f2bf(z);
  }
}

cudaError_t launch_quantize(int wquant, const uint16_t* w, int N, int K, void* codes, uint16_t* scales,
                            uint16_t* zeros, cudaStream_t s, const int32_t* perm) {
  if (N <= 0 || K <= 0) return cudaSuccess;
  if (wquant == FP_W_BF16) {
    return cudaMemcpyAsync(codes, w, (size_t)N * K * 2, cudaMemcpyDeviceToDevice, s);
  }
  if (wquant == FP_W_INT8) {
    return launch(quantize_int8_kernel, dim3(N), dim3(256), 0, s, w, K, (int8_t*)codes, scales);
  }
  long long warps = (long long)N * (K / 128);
  int blocks = (int)((warps + 7) / 8);
  return launch(quantize_int4_kernel, dim3(blocks), dim3(256), 0, s, w, N, K, (uint8_t*)codes, scales, zeros,
                wquant == FP_W_GPTQ4 ? perm : nullptr);
}

// ------------------------------------------------------------------ act order
// xp[m][j] = x[m][perm[j]]: the activations in a GPTQ4 matrix's act order,
// eight columns (one 16-byte store) per thread.  An entry of perm outside
// [0, K) reads as 0 and sets *err = 1.
__global__ void gather_cols_kernel(const uint16_t* __restrict__ x, int M, int K, const int32_t* __restrict__ perm,
                                   uint16_t* __restrict__ xp, int32_t* err) {
  pdl_trigger();
  pdl_wait();
  const long long units = (long long)M * (K / 8);
  bool bad = false;
  for (long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x; u < units;
       u += (long long)gridDim.x * blockDim.x) {
    const long long m = u / (K / 8);
    const int j0 = (int)(u % (K / 8)) * 8;
    const uint16_t* xr = x + m * K;
    uint32_t v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int k = perm[j0 + i];
      const bool in = (unsigned)k < (unsigned)K;
      bad |= !in;
      v[i] = in ? (uint32_t)xr[k] : 0u;
    }
    *reinterpret_cast<uint4*>(xp + m * K + j0) =
        make_uint4(v[0] | (v[1] << 16), v[2] | (v[3] << 16), v[4] | (v[5] << 16), v[6] | (v[7] << 16));
  }
  if (bad && err) atomicExch(err, 1);
}

// inv[perm[j]] = j; entries of perm outside [0, K) are skipped and set *err = 1
__global__ void invert_perm_kernel(const int32_t* __restrict__ perm, int K, int32_t* __restrict__ inv, int32_t* err) {
  pdl_trigger();
  pdl_wait();
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < K; j += gridDim.x * blockDim.x) {
    const int k = perm[j];
    if ((unsigned)k < (unsigned)K) inv[k] = j;
    else if (err) atomicExch(err, 1);
  }
}

cudaError_t launch_gather_cols(const uint16_t* x, int M, int K, const int32_t* perm, uint16_t* xp, int32_t* err,
                               cudaStream_t s) {
  if (M <= 0 || K <= 0) return cudaSuccess;
  const long long units = (long long)M * (K / 8);
  const int blocks = (int)std::min<long long>((units + 255) / 256, 152 * 8);
  return launch(gather_cols_kernel, dim3(blocks), dim3(256), 0, s, x, M, K, perm, xp, err);
}

cudaError_t launch_invert_perm(const int32_t* perm, int K, int32_t* inv, int32_t* err, cudaStream_t s) {
  if (K <= 0) return cudaSuccess;
  return launch(invert_perm_kernel, dim3(std::min((K + 255) / 256, 152 * 4)), dim3(256), 0, s, perm, K, inv, err);
}

}  // namespace fpk
