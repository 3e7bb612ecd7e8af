// Weight-only linear layers with the dequantisation fused into the product:
// y = x W^T, x bf16 [M][K], W bf16 / int8 per-channel / int4 group-128 (the
// INT8 and INT4 weight-only configurations, Sec. 3.2; formats in fp.h).
//
// Two kernels, chosen by the number of rows M of x:
//  * gemv_mma_kernel (M <= 64, decode): HBM-bound.  Each warp streams 16-row
//    tiles of codes with 16-byte non-allocating loads, turns them into bf16
//    MMA operands in registers (raw int8 codes, 128 + int4 codes), and runs
//    mma.sync m16n8k16 against x staged once per CTA in shared memory.
//    Scales are applied in fp32 (int8: per row in the epilogue; int4: per
//    128-group, s * (acc - (128 + z) * sum x)), so the weights enter exactly.
//    K is split across CTAs; the last CTA of a row block to finish sums the
//    partials and runs the epilogue (no spinning).
//  * gemv_kernel (fallback: larger M or a K that is not a multiple of the
//    MMA super-step): CUDA cores, one warp per output row.
#include <algorithm>

#include <cuda_fp16.h>

#include "common.cuh"
#include "kernels.cuh"

namespace fpk {

// Elements of K in one 16-byte chunk of codes.
template <int WQ>
struct WFmt;
template <>
struct WFmt<FP_W_BF16> { static constexpr int VE = 8; };
template <>
struct WFmt<FP_W_INT8> { static constexpr int VE = 16; };
template <>
struct WFmt<FP_W_INT4_G128> { static constexpr int VE = 32; };

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
      const uint32_t word = ww[h];  // elements 8h .. 8h+7; nibbles i and i+4 hold elements 2i and 2i+1
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float2 b = bf2x2f(xx[i]);
        const float lo = (float)((word >> (4 * i)) & 0xF) - zero;
        const float hi = (float)((word >> (4 * i + 16)) & 0xF) - zero;
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
  pdl_trigger();
  pdl_wait();
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
    case FP_EPI_STORE: return launch(gemv_kernel<WQ, MT, FP_EPI_STORE>, grid, dim3(256), 0, s, x, M, N, K, codes, scales, zeros, R, y);
    case FP_EPI_RESID: return launch(gemv_kernel<WQ, MT, FP_EPI_RESID>, grid, dim3(256), 0, s, x, M, N, K, codes, scales, zeros, R, y);
    case FP_EPI_SWIGLU: return launch(gemv_kernel<WQ, MT, FP_EPI_SWIGLU>, grid, dim3(256), 0, s, x, M, N, K, codes, scales, zeros, R, y);
    default: return launch(gemv_kernel<WQ, MT, FP_EPI_F32>, grid, dim3(256), 0, s, x, M, N, K, codes, scales, zeros, R, y);
  }
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


// =====================================================================
// Decode GEMV on tensor cores (mma.sync m16n8k16, fp32 accumulation)
// =====================================================================
// Thread (g = lane / 4, t = lane % 4) of a warp loads one 16-byte chunk of
// codes per row and super-step: KT consecutive k starting at t * KT.  Its
// k-slots of MMA k-step j are its local elements 4j .. 4j+3 (slots 2t, 2t+1
// <- 4j, 4j+1 and slots 2t+8, 2t+9 <- 4j+2, 4j+3); x uses the same map, so
// the contraction is unchanged.
//
// Operands: bf16 weights multiply bf16 x as they are.  int8 and int4 codes
// become fp16 by the 0x6400 exponent trick -- fp16(1152 + q) for int8,
// fp16(1024 + q) for int4, both exact -- and x is staged as fp16 (exact
// for |x| in the fp16 normal range; |x| >= 65504 is not supported).  The
// offsets are removed in fp32: int8 acc - 1152 * sum(x) over the CTA's K
// range, int4 per 128-group s * (acc - (1024 + z) * sum(x)).
template <int WQ>
struct MmaFmt;
template <>
struct MmaFmt<FP_W_BF16> { static constexpr int KT = 8; };
template <>
struct MmaFmt<FP_W_INT8> { static constexpr int KT = 16; };
template <>
struct MmaFmt<FP_W_INT4_G128> { static constexpr int KT = 32; };

constexpr int kGemvWarps = 8;  // warps per CTA; each owns one 16-row tile (two for SwiGLU: gate and up)

// 16-byte asynchronous global -> shared copy (L2 only), and its group fences.
FP_DEV void cp_async16(void* smem, const void* gmem) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s), "l"(gmem) : "memory");
}
FP_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
FP_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <bool F16>
FP_DEV void mma16816(float* c, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0, uint32_t b1) {
  if constexpr (F16) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  } else {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  }
}

FP_DEV uint32_t word_of(const uint4& w, int i) { return i == 0 ? w.x : i == 1 ? w.y : i == 2 ? w.z : w.w; }

// Thread-local elements 4j + 2h, 4j + 2h + 1 of a code chunk as an operand pair.
template <int WQ>
FP_DEV uint32_t apair(const uint4& w, int j, int h) {
  if constexpr (WQ == FP_W_BF16) {
    return word_of(w, 2 * j + h);
  } else if constexpr (WQ == FP_W_INT8) {
    // offset binary (q + 128) into the low byte of fp16 0x64xx = 1024 + (q + 128)
    const uint32_t word = word_of(w, j) ^ 0x80808080u;
    return __byte_perm(word, 0x64646464u, h ? 0x5342 : 0x5140);
  } else {
    // word j/2 holds elements 8(j/2) .. +7; nibbles i, i+4 hold elements 2i, 2i+1
    const uint32_t word = word_of(w, j >> 1);
    const int sh = 8 * (j & 1) + 4 * h;
    return ((word >> sh) & 0x000F000Fu) | 0x64006400u;  // fp16 1024 + q, both halves
  }
}

template <int WQ>
FP_DEV long long code_bytes(long long k) {
  return WQ == FP_W_BF16 ? 2 * k : WQ == FP_W_INT8 ? k : k / 2;
}

// x (bf16) -> MMA operand words: unchanged for bf16 weights, fp16 for codes.
template <int WQ>
FP_DEV uint4 x_operand(uint4 v) {
  if constexpr (WQ == FP_W_BF16) {
    return v;
  } else {
    uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = bf2x2f(w4[i]);
      const __half2 hh = __floats2half2_rn(f.x, f.y);
      w4[i] = *reinterpret_cast<const uint32_t*>(&hh);
    }
    return make_uint4(w4[0], w4[1], w4[2], w4[3]);
  }
}

template <int WQ>
FP_DEV float2 x_pair(uint32_t w) {
  if constexpr (WQ == FP_W_BF16) {
    return bf2x2f(w);
  } else {
    return __half22float2(*reinterpret_cast<const __half2*>(&w));
  }
}

// cp.async ring depth per warp: deeper for one tile, shallower for gate + up.
__host__ __device__ constexpr int gemv_stages(int tiles) { return tiles >= 2 ? 3 : 4; }

template <int WQ, int NT, int RT, int EPI>
__global__ void __launch_bounds__(kGemvWarps * 32) gemv_mma_kernel(const uint16_t* __restrict__ X, int M, int N, int K,
                                                       const void* __restrict__ codes,
                                                       const uint16_t* __restrict__ scales,
                                                       const uint16_t* __restrict__ zeros, const uint16_t* R,
                                                       void* Y, int ksplit, int splits, float* __restrict__ ws,
                                                       unsigned* __restrict__ counters) {
  constexpr int KT = MmaFmt<WQ>::KT, SUP = 4 * KT, KS = KT / 4, CH = KT / 8;
  constexpr bool F16 = WQ != FP_W_BF16;
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  constexpr int RTT = RT * NR;
  constexpr int NB = gemv_stages(RTT);  // ring stages per warp (NB - 1 in flight)
  extern __shared__ uint4 xs[];  // x of [kb, ke) in fragment order, then fp32 column sums
  __shared__ int s_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const int Nout = NR == 2 ? N / 2 : N;
  const int kb = blockIdx.y * ksplit;
  const int nsup = (min(K, kb + ksplit) - kb) / SUP;

  // ---- this warp's rows: tile rt covers rows (tile0 + rt) * 16 + g (+8); part r: gate / up
  const int tile0 = (blockIdx.x * kGemvWarps + warp) * RT;
  const uint8_t* wp[RTT][2];
  int rows[RTT][2];
#pragma unroll
  for (int rt = 0; rt < RT; ++rt)
#pragma unroll
    for (int r = 0; r < NR; ++r)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int row = (tile0 + rt) * 16 + g + 8 * h;
        const int rc = min(row, Nout - 1) + r * Nout;
        rows[rt * NR + r][h] = rc;
        wp[rt * NR + r][h] = (const uint8_t*)codes + code_bytes<WQ>((long long)rc * K + kb + t * KT);
      }
  pdl_trigger();
  // Weight chunks go through a per-warp ring in shared memory: each thread
  // copies its own 16-byte chunks with cp.async and later reads back only
  // those, so the ring needs no barrier.  The first stages go out before x
  // is staged.
  const int units = nsup * NT * CH * 32;
  const int xsum_entries = WQ == FP_W_BF16 ? 0 : (WQ == FP_W_INT8 ? 1 : nsup) * NT * 8;
  uint4* ring = xs + units + (xsum_entries + 3) / 4;
  auto slot = [&](int stage, int a, int h) { return ring + (((warp * NB + stage) * RTT + a) * 2 + h) * 32 + lane; };
#pragma unroll
  for (int b = 0; b < NB - 1; ++b) {
    if (b < nsup) {
#pragma unroll
      for (int a = 0; a < RTT; ++a) {
        cp_async16(slot(b, a, 0), wp[a][0] + b * 64);
        cp_async16(slot(b, a, 1), wp[a][1] + b * 64);
      }
    }
    cp_async_commit();
  }

  // weights are constant; everything below reads or writes the previous kernels' data
  pdl_wait();
  // ---- stage x rows 0 .. 8 NT - 1 (zero at and past M) as MMA operands:
  //      16-byte unit ((s NT + nt) CH + c) 32 + lane <- x[nt 8 + g][kb + s SUP + t KT + 8c .. +7]
  // and, for codes, the fp32 column sums of the staged operands: int8 over the
  // CTA's K range [8 NT], int4 per super-step (= one 128-group) [nsup][8 NT].
  float* xsum = reinterpret_cast<float*>(xs + units);
  if constexpr (F16) {
    for (int e = threadIdx.x; e < xsum_entries; e += blockDim.x) xsum[e] = 0.f;
    __syncthreads();
  }
  // units / 32 is a whole number, so every warp iterates with all 32 lanes
  for (int u = threadIdx.x; u < units; u += blockDim.x) {
    const int ln = u & 31, rest = u >> 5;
    const int c = rest % CH, snt = rest / CH, nt = snt % NT, s = snt / NT;
    const int m = nt * 8 + (ln >> 2);
    uint4 v = make_uint4(0, 0, 0, 0);
    if (m < M) v = x_operand<WQ>(ld_nc16(X + (long long)m * K + kb + s * SUP + (ln & 3) * KT + 8 * c));
    xs[u] = v;
    if constexpr (F16) {
      const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
      float sum = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = x_pair<WQ>(w4[i]);
        sum += f.x + f.y;
      }
      // the 4 lanes of one x row (same g) hold consecutive pieces of it
      sum += __shfl_xor_sync(0xffffffffu, sum, 1);
      sum += __shfl_xor_sync(0xffffffffu, sum, 2);
      if ((ln & 3) == 0) atomicAdd(&xsum[(WQ == FP_W_INT8 ? 0 : s * NT * 8) + m], sum);
    }
  }
  __syncthreads();
  const int groups = K / 128;

  float acc[RTT][NT][4];
#pragma unroll
  for (int a = 0; a < RTT; ++a)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) acc[a][nt][0] = acc[a][nt][1] = acc[a][nt][2] = acc[a][nt][3] = 0.f;

  for (int s = 0; s < nsup; ++s) {
    cp_async_wait<NB - 2>();  // this thread's copies of stage s have landed
    uint4 w[RTT][2];
#pragma unroll
    for (int a = 0; a < RTT; ++a) {
      w[a][0] = *slot(s % NB, a, 0);
      w[a][1] = *slot(s % NB, a, 1);
    }
    // refill the slot consumed one step ago with stage s + NB - 1
    const int sp = s + NB - 1;
    if (sp < nsup) {
#pragma unroll
      for (int a = 0; a < RTT; ++a) {
        cp_async16(slot(sp % NB, a, 0), wp[a][0] + sp * 64);
        cp_async16(slot(sp % NB, a, 1), wp[a][1] + sp * 64);
      }
    }
    cp_async_commit();
    float tmp[WQ == FP_W_INT4_G128 ? RTT : 1][NT][4];
    if constexpr (WQ == FP_W_INT4_G128) {
#pragma unroll
      for (int a = 0; a < RTT; ++a)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) tmp[a][nt][0] = tmp[a][nt][1] = tmp[a][nt][2] = tmp[a][nt][3] = 0.f;
    }
#pragma unroll
    for (int j = 0; j < KS; ++j) {
      uint32_t b0[NT], b1[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const uint4 xv = xs[((s * NT + nt) * CH + (j >> 1)) * 32 + lane];
        b0[nt] = (j & 1) ? xv.z : xv.x;
        b1[nt] = (j & 1) ? xv.w : xv.y;
      }
#pragma unroll
      for (int a = 0; a < RTT; ++a) {
        const uint32_t a0 = apair<WQ>(w[a][0], j, 0), a1 = apair<WQ>(w[a][1], j, 0);
        const uint32_t a2 = apair<WQ>(w[a][0], j, 1), a3 = apair<WQ>(w[a][1], j, 1);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          if constexpr (WQ == FP_W_INT4_G128) mma16816<F16>(tmp[a][nt], a0, a1, a2, a3, b0[nt], b1[nt]);
          else mma16816<F16>(acc[a][nt], a0, a1, a2, a3, b0[nt], b1[nt]);
        }
      }
    }
    if constexpr (WQ == FP_W_INT4_G128) {
      // acc += s * (sum (1024 + q) x - (1024 + z) sum x) over the group
      const int gi = (kb + s * SUP) / 128;
#pragma unroll
      for (int a = 0; a < RTT; ++a)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const long long si = (long long)rows[a][h] * groups + gi;
          const float sc = bf2f(scales[si]);
          const float zc = 1024.f + bf2f(zeros[si]);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int c = 0; c < 2; ++c) {
              const float xsm = xsum[s * NT * 8 + nt * 8 + 2 * t + c];
              acc[a][nt][2 * h + c] += sc * (tmp[a][nt][2 * h + c] - zc * xsm);
            }
        }
    }
  }
  cp_async_wait<0>();
  if constexpr (WQ == FP_W_INT8) {
    // remove the 1152 offset of the codes: acc - 1152 * sum x over this K range
#pragma unroll
    for (int a = 0; a < RTT; ++a)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[a][nt][i] -= 1152.f * xsum[nt * 8 + 2 * t + (i & 1)];
  }

  // ---- epilogue
  auto finish = [&](int m, int row, float v, float u) {
    if constexpr (WQ == FP_W_INT8) {
      v *= bf2f(scales[row]);
      if (NR == 2) u *= bf2f(scales[row + Nout]);
    }
    const long long o = (long long)m * Nout + row;
    if constexpr (EPI == FP_EPI_STORE) ((uint16_t*)Y)[o] = f2bf(v);
    else if constexpr (EPI == FP_EPI_RESID) ((uint16_t*)Y)[o] = f2bf(bf2f(R[o]) + v);
    else if constexpr (EPI == FP_EPI_SWIGLU) ((uint16_t*)Y)[o] = f2bf(silu(v) * u);
    else ((float*)Y)[o] = v;
  };
  if (splits == 1) {
#pragma unroll
    for (int rt = 0; rt < RT; ++rt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int row = (tile0 + rt) * 16 + g + 8 * (i >> 1);
          const int m = nt * 8 + 2 * t + (i & 1);
          if (row < Nout && m < M) finish(m, row, acc[rt * NR][nt][i], acc[rt * NR + NR - 1][nt][i]);
        }
    return;
  }
  // split-K: publish the partial, the last CTA of this row block reduces
#pragma unroll
  for (int rt = 0; rt < RT; ++rt)
#pragma unroll
    for (int r = 0; r < NR; ++r)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int row = (tile0 + rt) * 16 + g + 8 * (i >> 1);
          const int m = nt * 8 + 2 * t + (i & 1);
          if (row < Nout && m < M) ws[((long long)blockIdx.y * M + m) * N + row + r * Nout] = acc[rt * NR + r][nt][i];
        }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(&counters[blockIdx.x], 1u) == (unsigned)(splits - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int rows_cta = kGemvWarps * RT * 16;
  const int r0 = blockIdx.x * rows_cta;
  for (int idx = threadIdx.x; idx < M * rows_cta; idx += blockDim.x) {
    const int m = idx / rows_cta, row = r0 + idx % rows_cta;
    if (row >= Nout) continue;
    float v = 0.f, u = 0.f;
    for (int sp = 0; sp < splits; ++sp) {
      const float* p = ws + ((long long)sp * M + m) * N + row;
      v += __ldcg(p);
      if (NR == 2) u += __ldcg(p + Nout);
    }
    finish(m, row, v, u);
  }
  if (threadIdx.x == 0) counters[blockIdx.x] = 0u;
}

// ---------------------------------------------------------------- planning
struct GemvPlan {
  int NT, RT, ksplit, splits, blocks;
  size_t smem, ws;
};

static int mma_kt(int wq) { return wq == FP_W_BF16 ? 8 : wq == FP_W_INT8 ? 16 : 32; }

// Workspace = a fixed area of split-K ticket counters (zero at rest), then the
// fp32 partials.  The ticket area has the same size for every launch, so the
// partials of one launch never land on the counters of the next.
constexpr int kTicketSlots = 4096;
static size_t counter_bytes(int) { return (size_t)kTicketSlots * 4; }

// Rows per CTA are at least 64, so N <= 64 * kTicketSlots keeps one ticket per row block.
static bool mma_ok(int wq, int M, int N, int K) {
  return M >= 1 && M <= 64 && K % (4 * mma_kt(wq)) == 0 && N <= 64 * kTicketSlots;
}

static int sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        n <= 0)
      n = 152;
  }
  return n;
}

// occ = resident CTAs per SM of the chosen kernel (register limited).  The
// grid targets one full wave: blocks * splits close to SMs * occ.
static GemvPlan plan_gemv(int wq, int epi, int M, int N, int K, int occ) {
  GemvPlan p{};
  const int SUP = 4 * mma_kt(wq);
  p.NT = M <= 8 ? 1 : M <= 16 ? 2 : M <= 32 ? 4 : 8;
  p.RT = 1;
  const int nr = epi == FP_EPI_SWIGLU ? 2 : 1;
  const int Nout = nr == 2 ? N / 2 : N;
  p.blocks = (Nout + kGemvWarps * p.RT * 16 - 1) / (kGemvWarps * p.RT * 16);
  occ = std::max(1, std::min(occ, 8));
  // shared memory per CTA: the weight ring plus the x chunk, within 200 KiB per SM
  const int ring = kGemvWarps * gemv_stages(nr * p.RT) * nr * p.RT * 2 * 512;
  const int xbytes_per_k = p.NT * 8 * 2;
  const int smem_cap = std::max(8 * 1024, std::min(96 * 1024, 200 * 1024 / occ) - ring);
  const int kmax = std::max(SUP, (smem_cap / xbytes_per_k) / SUP * SUP);
  // whole waves: as many splits as fit in the resident slots (at least one)
  const int slots = sm_count() * occ;
  const int want = std::max(1, slots / p.blocks);
  int ks = (K + want - 1) / want;
  ks = (ks + SUP - 1) / SUP * SUP;
  ks = std::min(std::max(ks, SUP), kmax);
  p.ksplit = ks;
  p.splits = (K + ks - 1) / ks;
  const int nsup = ks / SUP;
  const size_t xsum_entries = wq == FP_W_BF16 ? 0 : (size_t)(wq == FP_W_INT8 ? 1 : nsup) * p.NT * 8;
  p.smem = (size_t)nsup * p.NT * mma_kt(wq) * 64 + (xsum_entries + 3) / 4 * 16 + ring;
  p.ws = p.splits > 1 ? counter_bytes(p.blocks) + (size_t)p.splits * M * N * 4 : 0;
  return p;
}

template <int WQ, int NT, int RT, int EPI>
static int gemv_occupancy() {
  static int occ = 0;
  if (!occ) {
    auto kern = gemv_mma_kernel<WQ, NT, RT, EPI>;
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, kGemvWarps * 32, 56 * 1024) != cudaSuccess ||
        occ <= 0)
      occ = 2;
    (void)cudaGetLastError();
  }
  return occ;
}

template <int WQ, int NT, int RT, int EPI>
static cudaError_t launch_mma_t(int wq, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                                const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* y, void* ws,
                                size_t ws_bytes, cudaStream_t s) {
  const GemvPlan p = plan_gemv(wq, epi, M, N, K, gemv_occupancy<WQ, NT, RT, EPI>());
  // never launch with less workspace than this plan writes
  if (p.ws > 0 && (!ws || ws_bytes < p.ws)) return cudaErrorInvalidValue;
  auto kern = gemv_mma_kernel<WQ, NT, RT, EPI>;  // dynamic shared memory limit set by gemv_occupancy
  if (p.smem > 200 * 1024) return cudaErrorInvalidValue;
  unsigned* counters = (unsigned*)ws;
  float* part = ws ? (float*)((char*)ws + counter_bytes(p.blocks)) : nullptr;
  dim3 grid(p.blocks, p.splits);
  return launch(kern, grid, dim3(kGemvWarps * 32), p.smem, s, x, M, N, K, codes, scales, zeros, R, y, p.ksplit,
                p.splits, part, counters);
}

template <int WQ, int EPI>
static cudaError_t launch_mma_e(int wq, const uint16_t* x, int M, int N, int K, const void* codes,
                                const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* y, void* ws,
                                size_t ws_bytes, cudaStream_t s) {
  const GemvPlan p = plan_gemv(wq, EPI, M, N, K, 1);  // NT and RT do not depend on occupancy
#define FP_MMA_CASE(nt, rt) \
  if (p.NT == nt && p.RT == rt)  \
    return launch_mma_t<WQ, nt, rt, EPI>(wq, EPI, x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s);
  FP_MMA_CASE(1, 1)
  FP_MMA_CASE(2, 1)
  FP_MMA_CASE(4, 1)
  FP_MMA_CASE(8, 1)
#undef FP_MMA_CASE
  return cudaErrorInvalidValue;
}

template <int WQ>
static cudaError_t launch_mma(int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                              const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* y, void* ws,
                              size_t ws_bytes, cudaStream_t s) {
  switch (epi) {
    case FP_EPI_STORE: return launch_mma_e<WQ, FP_EPI_STORE>(WQ, x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s);
    case FP_EPI_RESID: return launch_mma_e<WQ, FP_EPI_RESID>(WQ, x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s);
    case FP_EPI_SWIGLU: return launch_mma_e<WQ, FP_EPI_SWIGLU>(WQ, x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s);
    default: return launch_mma_e<WQ, FP_EPI_F32>(WQ, x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s);
  }
}

// Workspace of one linear launch: the ticket area, then either split-K
// partials (decode GEMV) or the bf16 expansion of quantised weights (prefill
// GEMM).  The ticket area is never written by the prefill path.
size_t linear_ws_bytes(int wquant, int M, int N, int K) {
  if (M > 64 && gemm_tc_ok(M, N, K)) {
    const size_t w = gemm_tc_ws_bytes(wquant, N, K);
    return w ? counter_bytes(0) + w : 0;
  }
  if (!mma_ok(wquant, M, N, K)) return 0;
  // splits grow with occupancy, so the plan at the planner's cap (8) bounds every launch
  size_t a = plan_gemv(wquant, FP_EPI_STORE, M, N, K, 8).ws;
  size_t b = N % 2 == 0 ? plan_gemv(wquant, FP_EPI_SWIGLU, M, N, K, 8).ws : 0;
  return std::max(a, b);
}

size_t linear_ws_bytes_upto(int wquant, int max_m, int N, int K) {
  size_t w = 0;
  for (int m = 1; m <= std::min(max_m, 64); ++m) w = std::max(w, linear_ws_bytes(wquant, m, N, K));
  if (max_m > 64) w = std::max(w, linear_ws_bytes(wquant, max_m, N, K));
  return w;
}

cudaError_t launch_linear(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                          const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                          void* ws, size_t ws_bytes, cudaStream_t s, int32_t* err) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  if (M > 64 && gemm_tc_ok(M, N, K)) {
    const size_t need = linear_ws_bytes(wquant, M, N, K);
    if (need > 0 && (!ws || ws_bytes < need)) return cudaErrorInvalidValue;
    void* scratch = need ? (char*)ws + counter_bytes(0) : nullptr;
    return launch_gemm_tc(wquant, epi, x, M, N, K, codes, scales, zeros, residual, y, scratch,
                          need ? ws_bytes - counter_bytes(0) : 0, err, s);
  }
  if (mma_ok(wquant, M, N, K)) {
    switch (wquant) {
      case FP_W_BF16: return launch_mma<FP_W_BF16>(epi, x, M, N, K, codes, scales, zeros, residual, y, ws, ws_bytes, s);
      case FP_W_INT8: return launch_mma<FP_W_INT8>(epi, x, M, N, K, codes, scales, zeros, residual, y, ws, ws_bytes, s);
      default: return launch_mma<FP_W_INT4_G128>(epi, x, M, N, K, codes, scales, zeros, residual, y, ws, ws_bytes, s);
    }
  }
  switch (wquant) {
    case FP_W_BF16: return launch_gemv<FP_W_BF16>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
    case FP_W_INT8: return launch_gemv<FP_W_INT8>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
    default: return launch_gemv<FP_W_INT4_G128>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
  }
}

}  // namespace fpk
