// Weight-only linear layers with the dequantisation fused into the product:
// y = x W^T, x bf16 [M][K], W bf16 / int8 per-channel / int4 group-128 (the
// INT8 and INT4 weight-only configurations, Sec. 3.2; formats in fp.h).
//
// This file holds the memory-bound decode GEMV: a warp owns one output row
// (two for SwiGLU: gate row n and up row n + N/2), streams the row's codes
// with 16-byte non-allocating loads, dequantises in registers and reduces
// over the warp; up to MT rows of x share each weight load.
#include "common.cuh"
#include "kernels.cuh"

namespace fpk {

template <int WQ>
struct WFmt;
template <>
struct WFmt<FP_W_BF16> { static constexpr int VE = 8;  static constexpr int RB = 2; };  // elements / 16 B chunk, row bytes per 1 element x RB/2
template <>
struct WFmt<FP_W_INT8> { static constexpr int VE = 16; static constexpr int RB = 1; };
template <>
struct WFmt<FP_W_INT4_G128> { static constexpr int VE = 32; static constexpr int RB = 0; };

// Row pointer of the codes of output row n.
template <int WQ>
FP_DEV const uint8_t* code_row(const void* codes, long long n, int K) {
  if (WQ == FP_W_BF16) return (const uint8_t*)codes + n * K * 2;
  if (WQ == FP_W_INT8) return (const uint8_t*)codes + n * K;
  return (const uint8_t*)codes + n * (K / 2);
}

// Dot of one 16-byte weight chunk with VE consecutive x values (bf16).
// Returns the partial sum in the weight's code domain:
//   bf16: sum w x;  int8: sum q x (scale applied later);  int4: sum (q - z) x.
template <int WQ>
FP_DEV float chunk_dot(const uint4& w, const uint16_t* xp, float zero) {
  const uint4* xv = reinterpret_cast<const uint4*>(xp);
  float acc = 0.f;
  if constexpr (WQ == FP_W_BF16) {
    uint4 x = ld_nc16(xv);
    const uint32_t ww[4] = {w.x, w.y, w.z, w.w}, xx[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 a = bf2x2f(ww[i]), b = bf2x2f(xx[i]);
      acc += a.x * b.x + a.y * b.y;
    }
  } else if constexpr (WQ == FP_W_INT8) {
    const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      uint4 x = ld_nc16(xv + h);
      const uint32_t xx[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t word = ww[2 * h + (i >> 1)];
        const int sh = 16 * (i & 1);
        float2 b = bf2x2f(xx[i]);
        acc += (float)(int8_t)((word >> sh) & 0xFF) * b.x + (float)(int8_t)((word >> (sh + 8)) & 0xFF) * b.y;
      }
    }
  } else {
    const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      uint4 x = ld_nc16(xv + h);
      const uint32_t xx[4] = {x.x, x.y, x.z, x.w};
      const uint32_t word = ww[h];  // 8 nibbles = elements 8h .. 8h+7
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float2 b = bf2x2f(xx[i]);
        const float lo = (float)((word >> (8 * i)) & 0xF) - zero;
        const float hi = (float)((word >> (8 * i + 4)) & 0xF) - zero;
        acc += lo * b.x + hi * b.y;
      }
    }
  }
  return acc;
}

template <int WQ, int MT, int EPI>
__global__ void __launch_bounds__(256) gemv_kernel(const uint16_t* __restrict__ X, int M, int N, int K,
                                                   const void* __restrict__ codes, const uint16_t* __restrict__ scales,
                                                   const uint16_t* __restrict__ zeros,
                                                   const uint16_t* __restrict__ R, void* __restrict__ Y) {
  constexpr int VE = WFmt<WQ>::VE;
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Nout = EPI == FP_EPI_SWIGLU ? N / 2 : N;
  const int n = blockIdx.y * 8 + warp;
  const int m0 = blockIdx.x * MT;
  if (n >= Nout) return;
  const int chunks = K / VE;
  const int groups = K / 128;
  float acc[NR][MT];
#pragma unroll
  for (int r = 0; r < NR; ++r)
#pragma unroll
    for (int m = 0; m < MT; ++m) acc[r][m] = 0.f;
  const int mcount = min(MT, M - m0);
#pragma unroll 2
  for (int c = lane; c < chunks; c += 32) {
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      const long long row = n + (long long)r * Nout;
      const uint4 w = ld_stream16(code_row<WQ>(codes, row, K) + (long long)c * 16);
      float sc = 1.f, zp = 0.f;
      if constexpr (WQ == FP_W_INT4_G128) {
        const int g = (c * VE) / 128;
        sc = bf2f(scales[row * groups + g]);
        zp = bf2f(zeros[row * groups + g]);
      }
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        if (m < mcount) {
          const float d = chunk_dot<WQ>(w, X + (long long)(m0 + m) * K + (long long)c * VE, zp);
          acc[r][m] += WQ == FP_W_INT4_G128 ? sc * d : d;
        }
      }
    }
  }
#pragma unroll
  for (int r = 0; r < NR; ++r)
#pragma unroll
    for (int m = 0; m < MT; ++m) acc[r][m] = warp_sum(acc[r][m]);
  if (lane < mcount) {
    // every lane holds every sum; lane m writes row m0 + m
    float v[NR];
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      float a = 0.f;
#pragma unroll
      for (int m = 0; m < MT; ++m) a = (m == lane) ? acc[r][m] : a;
      if constexpr (WQ == FP_W_INT8) a *= bf2f(scales[n + (long long)r * Nout]);
      v[r] = a;
    }
    const long long o = (long long)(m0 + lane) * Nout + n;
    if constexpr (EPI == FP_EPI_STORE) {
      ((uint16_t*)Y)[o] = f2bf(v[0]);
    } else if constexpr (EPI == FP_EPI_RESID) {
      ((uint16_t*)Y)[o] = f2bf(bf2f(R[o]) + v[0]);
    } else if constexpr (EPI == FP_EPI_SWIGLU) {
      ((uint16_t*)Y)[o] = f2bf(silu(v[0]) * v[NR - 1]);
    } else {
      ((float*)Y)[o] = v[0];
    }
  }
}

template <int WQ, int MT>
static cudaError_t launch_gemv_mt(int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                                  const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* y,
                                  cudaStream_t s) {
  const int Nout = epi == FP_EPI_SWIGLU ? N / 2 : N;
  // M tiles on x (fastest) so CTAs that share weight rows run together.
  dim3 grid((M + MT - 1) / MT, (Nout + 7) / 8);
  switch (epi) {
    case FP_EPI_STORE: gemv_kernel<WQ, MT, FP_EPI_STORE><<<grid, 256, 0, s>>>(x, M, N, K, codes, scales, zeros, R, y); break;
    case FP_EPI_RESID: gemv_kernel<WQ, MT, FP_EPI_RESID><<<grid, 256, 0, s>>>(x, M, N, K, codes, scales, zeros, R, y); break;
    case FP_EPI_SWIGLU: gemv_kernel<WQ, MT, FP_EPI_SWIGLU><<<grid, 256, 0, s>>>(x, M, N, K, codes, scales, zeros, R, y); break;
    default: gemv_kernel<WQ, MT, FP_EPI_F32><<<grid, 256, 0, s>>>(x, M, N, K, codes, scales, zeros, R, y); break;
  }
  return cudaGetLastError();
}

template <int WQ>
static cudaError_t launch_gemv(int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                               const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* y,
                               cudaStream_t s) {
  if (M <= 1) return launch_gemv_mt<WQ, 1>(epi, x, M, N, K, codes, scales, zeros, R, y, s);
  if (M <= 2) return launch_gemv_mt<WQ, 2>(epi, x, M, N, K, codes, scales, zeros, R, y, s);
  if (M <= 4) return launch_gemv_mt<WQ, 4>(epi, x, M, N, K, codes, scales, zeros, R, y, s);
  return launch_gemv_mt<WQ, 8>(epi, x, M, N, K, codes, scales, zeros, R, y, s);
}

size_t linear_ws_bytes(int wquant, int M, int N, int K) {
  (void)wquant; (void)M; (void)N; (void)K;
  return 0;
}

cudaError_t launch_linear(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                          const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                          void* ws, cudaStream_t s) {
  (void)ws;
  if (M <= 0 || N <= 0) return cudaSuccess;
  switch (wquant) {
    case FP_W_BF16: return launch_gemv<FP_W_BF16>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
    case FP_W_INT8: return launch_gemv<FP_W_INT8>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
    default: return launch_gemv<FP_W_INT4_G128>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
  }
}

}  // namespace fpk
