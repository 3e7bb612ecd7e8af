// Weight-only linear layers with the dequantisation fused into the product:
// y = x W^T, x bf16 [M][K], W bf16 / int8 per-channel / int4 group-128 (the
// INT8 and INT4 weight-only configurations, Sec. 3.2; formats in fp.h).
//
// Two kernels, chosen by the number of rows M of x:
//  * gemv_mma_kernel (M <= 64, decode): HBM-bound.  Each warp streams 16-row
//    tiles of codes through a per-thread cp.async ring, turns them into MMA
//    operands in registers, and runs mma.sync m16n8k16 against x staged
//    once per window in shared memory.  bf16 weights enter as they are; int8
//    and int4 codes become fp16(1152 + q) and fp16(1024 + q) by the exponent
//    trick (exact), with x staged as fp16.  Offsets and scales are removed in
//    fp32 (int8: acc - 1152 sum x, times the row scale in the epilogue; int4:
//    per 128-group, s (acc - (1024 + z) sum x)), so the weights enter exactly.
//    The (row block, K step) work is cut into equal contiguous ranges, one
//    per resident CTA; a row block shared by several CTAs is finished by the
//    last of them from fp32 partials (no spinning).
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
// for |x| in the fp16 normal range; smaller values become fp16 subnormals,
// and an |x| that rounds beyond 65504 becomes inf and sets the error word to
// 3, which the runtime reports).  The offsets are removed in fp32: int8
// acc - 1152 * sum(x) over the CTA's K range, int4 per 128-group
// s * (acc - (1024 + z) * sum(x)).
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

// cp.async ring depth per warp (NB - 1 stages in flight): deeper for one
// tile, shallower for gate + up.
__host__ __device__ constexpr int gemv_stages(int tiles) { return tiles >= 2 ? 3 : 6; }

// The work of one launch is the sequence of (row block, super-step) pairs,
// row block major: blocks x S with S = K / super-step.  CTA c of C takes the
// contiguous range [c total / C, (c+1) total / C), so every CTA streams the
// same number of weight bytes whatever N and K are, and one wave of
// resident CTAs covers the launch.  A range crosses row blocks: the CTA
// accumulates each block's part separately and, where a block is shared by
// several CTAs, the last to finish sums their fp32 partials in CTA order
// (deterministic) and runs the epilogue.
FP_DEV long long gemv_cta_of(long long i, long long C, long long total) { return ((i + 1) * C - 1) / total; }

template <int WQ, int NT, int EPI>
__global__ void __launch_bounds__(kGemvWarps * 32) gemv_mma_kernel(const uint16_t* __restrict__ X, int M, int N, int K,
                                                       const void* __restrict__ codes,
                                                       const uint16_t* __restrict__ scales,
                                                       const uint16_t* __restrict__ zeros, const uint16_t* R,
                                                       void* Y, long long total, int S, int W,
                                                       float* __restrict__ ws, unsigned* __restrict__ counters,
                                                       int32_t* err) {
  constexpr int KT = MmaFmt<WQ>::KT, SUP = 4 * KT, KS = KT / 4, CH = KT / 8;
  constexpr bool F16 = WQ != FP_W_BF16;
  constexpr bool G128 = WQ == FP_W_INT4_G128;
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  constexpr int NB = gemv_stages(NR);
  constexpr int ROWS = kGemvWarps * 16;  // rows of a block
  extern __shared__ uint4 smem[];        // weight ring, then the x window, then its fp32 column sums
  __shared__ int s_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const int Nout = NR == 2 ? N / 2 : N;
  const int groups = K / 128;
  const long long C = gridDim.x, c = blockIdx.x;
  const long long begin = c * total / C, end = (c + 1) * total / C;
  const int L = (int)(end - begin);

  uint4* ring = smem;
  uint4* xs = smem + kGemvWarps * NB * NR * 2 * 32;
  float* xsum = reinterpret_cast<float*>(xs + W * NT * CH * 32);
  auto slot = [&](int stage, int r, int h) { return ring + (((warp * NB + stage) * NR + r) * 2 + h) * 32 + lane; };
  auto row_of = [&](int blk, int h) { return blk * ROWS + warp * 16 + g + 8 * h; };

  // ---- weight ring: each thread copies its own 16-byte chunks with cp.async
  // and later reads back only those, so the ring needs no barrier.  Stage q
  // of this CTA is super-step (begin + q) % S of row block (begin + q) / S.
  int pf_blk = (int)(begin / S), pf_ss = (int)(begin % S);
  const uint8_t* pw[NR][2];
  auto set_rows = [&](int blk) {
#pragma unroll
    for (int r = 0; r < NR; ++r)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int rc = min(row_of(blk, h), Nout - 1) + r * Nout;
        pw[r][h] = (const uint8_t*)codes + code_bytes<WQ>((long long)rc * K + t * KT);
      }
  };
  set_rows(pf_blk);
  auto issue = [&](int q) {  // called for q = 0, 1, 2, ... in order
    if (q < L) {
#pragma unroll
      for (int r = 0; r < NR; ++r)
#pragma unroll
        for (int h = 0; h < 2; ++h) cp_async16(slot(q % NB, r, h), pw[r][h] + pf_ss * 64);
      if (++pf_ss == S) {
        pf_ss = 0;
        set_rows(++pf_blk);  // row pointers are clamped, so a block past the end is harmless
      }
    }
    cp_async_commit();
  };
  pdl_trigger();
  // weights are constant: the first stages go out before waiting on the producer of x
#pragma unroll
  for (int q = 0; q < NB - 1; ++q) issue(q);
  pdl_wait();

  float acc[NR][NT][4];
  auto zero_acc = [&]() {
#pragma unroll
    for (int r = 0; r < NR; ++r)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) acc[r][nt][0] = acc[r][nt][1] = acc[r][nt][2] = acc[r][nt][3] = 0.f;
  };
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
  zero_acc();

  long long cur = begin;
  int q = 0;
  while (cur < end) {
    const int b = (int)(cur / S), s0 = (int)(cur % S);
    const long long seg_end = min(end, (long long)(b + 1) * S);
    const int wlen = (int)min((long long)W, seg_end - cur);

    // ---- stage x for super-steps s0 .. s0 + wlen - 1 of K as MMA operands:
    //      16-byte unit ((l NT + nt) CH + c) 32 + lane <- x[nt 8 + g][(s0 + l) SUP + t KT + 8c .. +7]
    // (zero at and past M) and, for codes, the fp32 column sums of the staged
    // operands: int8 over the window [8 NT], int4 per super-step (= one
    // 128-group) [wlen][8 NT].
    const int units = wlen * NT * CH * 32;
    const int nsum = F16 ? (G128 ? wlen : 1) * NT * 8 : 0;
    __syncthreads();  // the previous window is consumed
    for (int e = threadIdx.x; e < nsum; e += blockDim.x) xsum[e] = 0.f;
    if constexpr (F16) __syncthreads();
    constexpr int XU = 4;  // independent x loads in flight per thread
    // units is a multiple of 32, so the lanes of a warp agree on u < units
    for (int u0 = threadIdx.x; u0 < units; u0 += XU * blockDim.x) {
      uint4 v[XU];
#pragma unroll
      for (int i = 0; i < XU; ++i) {
        const int u = u0 + i * blockDim.x;
        const int ln = u & 31, rest = u >> 5;
        const int cc = rest % CH, lnt = rest / CH, nt = lnt % NT, l = lnt / NT;
        const int m = nt * 8 + (ln >> 2);
        v[i] = make_uint4(0, 0, 0, 0);
        if (u < units && m < M) v[i] = ld_nc16(X + (long long)m * K + (s0 + l) * SUP + (ln & 3) * KT + 8 * cc);
      }
#pragma unroll
      for (int i = 0; i < XU; ++i) {
        const int u = u0 + i * blockDim.x;
        if (u < units) {
          const int ln = u & 31, rest = u >> 5;
          const int lnt = rest / CH, nt = lnt % NT, l = lnt / NT;
          const uint4 xo = x_operand<WQ>(v[i]);
          xs[u] = xo;
          if constexpr (F16) {
            const uint32_t w4[4] = {xo.x, xo.y, xo.z, xo.w};
            float sum = 0.f;
            bool over = false;
#pragma unroll
            for (int p = 0; p < 4; ++p) {
              const float2 f = x_pair<WQ>(w4[p]);
              sum += f.x + f.y;
              over |= isinf(f.x) || isinf(f.y);
            }
            if (over && err) atomicExch(err, 3);  // x outside the fp16 range: the output is invalid
            // the 4 lanes of one x row (same g) hold consecutive pieces of it
            sum += __shfl_xor_sync(0xffffffffu, sum, 1);
            sum += __shfl_xor_sync(0xffffffffu, sum, 2);
            if ((ln & 3) == 0) atomicAdd(&xsum[(G128 ? l * NT * 8 : 0) + nt * 8 + (ln >> 2)], sum);
          }
        }
      }
    }
    __syncthreads();

    // ---- the window's super-steps
    for (int l = 0; l < wlen; ++l, ++q) {
      cp_async_wait<NB - 2>();  // this thread's copies of stage q have landed
      uint4 w[NR][2];
#pragma unroll
      for (int r = 0; r < NR; ++r) {
        w[r][0] = *slot(q % NB, r, 0);
        w[r][1] = *slot(q % NB, r, 1);
      }
      issue(q + NB - 1);  // refills the slot consumed one step ago
      float sz[G128 ? NR : 1][2][2];
      if constexpr (G128) {
#pragma unroll
        for (int r = 0; r < NR; ++r)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const long long si = (long long)(min(row_of(b, h), Nout - 1) + r * Nout) * groups + s0 + l;
            sz[r][h][0] = bf2f(__ldg(scales + si));
            sz[r][h][1] = 1024.f + bf2f(__ldg(zeros + si));
          }
      }
      float tmp[G128 ? NR : 1][NT][4];
      if constexpr (G128) {
#pragma unroll
        for (int r = 0; r < NR; ++r)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) tmp[r][nt][0] = tmp[r][nt][1] = tmp[r][nt][2] = tmp[r][nt][3] = 0.f;
      }
#pragma unroll
      for (int j = 0; j < KS; ++j) {
        uint32_t b0[NT], b1[NT];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          const uint4 xv = xs[((l * NT + nt) * CH + (j >> 1)) * 32 + lane];
          b0[nt] = (j & 1) ? xv.z : xv.x;
          b1[nt] = (j & 1) ? xv.w : xv.y;
        }
#pragma unroll
        for (int r = 0; r < NR; ++r) {
          const uint32_t a0 = apair<WQ>(w[r][0], j, 0), a1 = apair<WQ>(w[r][1], j, 0);
          const uint32_t a2 = apair<WQ>(w[r][0], j, 1), a3 = apair<WQ>(w[r][1], j, 1);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            if constexpr (G128) mma16816<F16>(tmp[r][nt], a0, a1, a2, a3, b0[nt], b1[nt]);
            else mma16816<F16>(acc[r][nt], a0, a1, a2, a3, b0[nt], b1[nt]);
          }
        }
      }
      if constexpr (G128) {
        // acc += s * (sum (1024 + q) x - (1024 + z) sum x) over the group
#pragma unroll
        for (int r = 0; r < NR; ++r)
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
              for (int cc = 0; cc < 2; ++cc) {
                const float xsm = xsum[l * NT * 8 + nt * 8 + 2 * t + cc];
                acc[r][nt][2 * h + cc] += sz[r][h][0] * (tmp[r][nt][2 * h + cc] - sz[r][h][1] * xsm);
              }
      }
    }
    if constexpr (WQ == FP_W_INT8) {
      // remove the 1152 offset of the codes: acc - 1152 * sum x over the window
#pragma unroll
      for (int r = 0; r < NR; ++r)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[r][nt][i] -= 1152.f * xsum[nt * 8 + 2 * t + (i & 1)];
    }
    cur += wlen;
    if (cur < seg_end) continue;

    // ---- row block b is done for this CTA
    const long long c0 = gemv_cta_of((long long)b * S, C, total);
    const long long c1 = gemv_cta_of((long long)(b + 1) * S - 1, C, total);
    if (c0 == c1) {
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int row = row_of(b, i >> 1);
          const int m = nt * 8 + 2 * t + (i & 1);
          if (row < Nout && m < M) finish(m, row, acc[0][nt][i], acc[NR - 1][nt][i]);
        }
    } else {
      // partial slot b + c: distinct for every (block, CTA) pair that meets
      float* part = ws + (size_t)(b + c) * M * NR * ROWS;
#pragma unroll
      for (int r = 0; r < NR; ++r)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int lr = warp * 16 + g + 8 * (i >> 1);
            const int m = nt * 8 + 2 * t + (i & 1);
            if (m < M) part[((long long)m * NR + r) * ROWS + lr] = acc[r][nt][i];
          }
      __threadfence();
      __syncthreads();
      if (threadIdx.x == 0) s_last = atomicAdd(&counters[b], 1u) == (unsigned)(c1 - c0);
      __syncthreads();
      if (s_last) {
        __threadfence();
        // four rows per thread; the partial loads of several CTAs are in flight together
        for (int idx = threadIdx.x; idx < M * (ROWS / 4); idx += blockDim.x) {
          const int m = idx / (ROWS / 4), lr = (idx % (ROWS / 4)) * 4;
          const size_t slot_f = (size_t)M * NR * ROWS;
          const float* p0 = ws + (size_t)(b + c0) * slot_f + (size_t)m * NR * ROWS + lr;
          float4 v = make_float4(0.f, 0.f, 0.f, 0.f), u = v;
          const int cnt = (int)(c1 - c0) + 1;
#pragma unroll 4
          for (int cc = 0; cc < cnt; ++cc) {
            const float4 a = __ldcg(reinterpret_cast<const float4*>(p0 + (size_t)cc * slot_f));
            v.x += a.x, v.y += a.y, v.z += a.z, v.w += a.w;
            if (NR == 2) {
              const float4 e = __ldcg(reinterpret_cast<const float4*>(p0 + (size_t)cc * slot_f + ROWS));
              u.x += e.x, u.y += e.y, u.z += e.z, u.w += e.w;
            }
          }
          const float vv[4] = {v.x, v.y, v.z, v.w}, uu[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int row = b * ROWS + lr + e;
            if (row < Nout) finish(m, row, vv[e], uu[e]);
          }
        }
        if (threadIdx.x == 0) counters[b] = 0u;
      }
    }
    zero_acc();
  }
  cp_async_wait<0>();
}

// ---------------------------------------------------------------- planning
struct GemvPlan {
  int NT, ctas, S, W, blocks;
  long long total;
  size_t smem, ws;
};

static int mma_kt(int wq) { return wq == FP_W_BF16 ? 8 : wq == FP_W_INT8 ? 16 : 32; }

// Workspace = a fixed area of ticket counters (zero at rest), then the fp32
// partials.  The ticket area has the same size for every launch, so the
// partials of one launch never land on the counters of the next.
constexpr int kTicketSlots = kLinTicketSlots;
static size_t counter_bytes(int) { return (size_t)kTicketSlots * 4; }

// One ticket per 128-row block.
static bool mma_ok(int wq, int M, int N, int K) {
  return M >= 1 && M <= 64 && K % (4 * mma_kt(wq)) == 0 && N <= kGemvWarps * 16 * kTicketSlots;
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

static int gemv_nt(int M) { return M <= 8 ? 1 : M <= 16 ? 2 : M <= 32 ? 4 : 8; }

// Shared-memory limits of a kernel: per CTA (dynamic) and per SM.
struct SmemLimits {
  int per_cta_dyn;  // opt-in maximum minus the kernel's static shared memory
  int per_sm;       // usable by CTAs on one SM
  int static_bytes;
};

// occ_max = CTAs per SM the kernel's registers allow.  The plan takes the
// most CTAs per SM whose shared memory (ring + an x window of at least a
// third of one CTA's range, up to a whole row block) fits, and one wave of
// CTAs.
static GemvPlan plan_gemv(int wq, int epi, int M, int N, int K, int occ_max, const SmemLimits& lim) {
  GemvPlan p{};
  const int SUP = 4 * mma_kt(wq);
  const int NT = gemv_nt(M);
  const int nr = epi == FP_EPI_SWIGLU ? 2 : 1;
  const int Nout = nr == 2 ? N / 2 : N;
  p.NT = NT;
  p.blocks = (Nout + kGemvWarps * 16 - 1) / (kGemvWarps * 16);
  p.S = K / SUP;
  p.total = (long long)p.blocks * p.S;
  const int ring = kGemvWarps * gemv_stages(nr) * nr * 2 * 512;
  const int per_ss = NT * SUP * 16 + (wq == FP_W_INT4_G128 ? NT * 8 * 4 : 0);  // x operands (+ int4 group sums)
  const int fixed = wq == FP_W_INT8 ? NT * 8 * 4 : 0;                           // int8 window sums
  const int sms = sm_count();
  occ_max = std::max(1, std::min(occ_max, 8));
  int best_occ = 0, best_w = 0;
  for (int occ = occ_max; occ >= 1; --occ) {
    const int budget = std::min(lim.per_cta_dyn, lim.per_sm / occ - 1024 - lim.static_bytes) - 16;
    const int wmax = (budget - ring - fixed) / per_ss;
    if (wmax < 1) continue;
    const long long C = std::min<long long>(p.total, (long long)occ * sms);
    const long long need = std::min<long long>((p.total + C - 1) / C, p.S);
    if (wmax > best_w) {
      best_w = wmax;
      best_occ = occ;
    }
    if (3LL * wmax >= need) {  // at most three x windows for the longest piece of a row block
      best_occ = occ;
      best_w = wmax;
      break;
    }
  }
  if (best_occ == 0) return p;  // ctas == 0: no plan
  p.ctas = (int)std::min<long long>(p.total, (long long)best_occ * sms);
  p.W = std::min(best_w, p.S);
  p.smem = (size_t)ring + (size_t)p.W * NT * SUP * 16 +
           (size_t)(wq == FP_W_INT4_G128 ? p.W : (wq == FP_W_INT8 ? 1 : 0)) * NT * 8 * 4;
  p.ws = counter_bytes(p.blocks) + (size_t)(p.blocks + p.ctas) * M * nr * kGemvWarps * 16 * 4;
  return p;
}

static int max_smem_optin() {
  static int v = 0;
  if (!v) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess || v <= 0)
      v = 227 * 1024;
  }
  return v;
}

static int smem_per_sm() {
  static int v = 0;
  if (!v) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) != cudaSuccess || v <= 0)
      v = 228 * 1024;
  }
  return v;
}

// CTAs per SM the kernel's registers allow, and its shared-memory limits;
// lifts the kernel's dynamic shared memory limit to the opt-in maximum.
template <int WQ, int NT, int EPI>
static int gemv_occupancy(SmemLimits* lim) {
  static int occ = 0;
  static SmemLimits l{};
  if (!occ) {
    auto kern = gemv_mma_kernel<WQ, NT, EPI>;
    cudaFuncAttributes fa{};
    int st = cudaFuncGetAttributes(&fa, kern) == cudaSuccess ? (int)fa.sharedSizeBytes : 64;
    l.static_bytes = st;
    l.per_cta_dyn = max_smem_optin() - st;
    l.per_sm = smem_per_sm();
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, l.per_cta_dyn);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, kGemvWarps * 32, 0) != cudaSuccess || occ <= 0)
      occ = 2;
    (void)cudaGetLastError();
  }
  *lim = l;
  return occ;
}

template <int WQ, int NT, int EPI>
static GemvPlan plan_t(int M, int N, int K) {
  SmemLimits lim{};
  const int occ = gemv_occupancy<WQ, NT, EPI>(&lim);
  return plan_gemv(WQ, EPI, M, N, K, occ, lim);
}

template <int WQ, int EPI>
static GemvPlan plan_e(int M, int N, int K) {
  switch (gemv_nt(M)) {
    case 1: return plan_t<WQ, 1, EPI>(M, N, K);
    case 2: return plan_t<WQ, 2, EPI>(M, N, K);
    case 4: return plan_t<WQ, 4, EPI>(M, N, K);
    default: return plan_t<WQ, 8, EPI>(M, N, K);
  }
}

template <int WQ>
static GemvPlan plan_w(int epi, int M, int N, int K) {
  switch (epi) {
    case FP_EPI_STORE: return plan_e<WQ, FP_EPI_STORE>(M, N, K);
    case FP_EPI_RESID: return plan_e<WQ, FP_EPI_RESID>(M, N, K);
    case FP_EPI_SWIGLU: return plan_e<WQ, FP_EPI_SWIGLU>(M, N, K);
    default: return plan_e<WQ, FP_EPI_F32>(M, N, K);
  }
}

// The plan a launch of this shape uses.
static GemvPlan plan_for(int wq, int epi, int M, int N, int K) {
  switch (wq) {
    case FP_W_BF16: return plan_w<FP_W_BF16>(epi, M, N, K);
    case FP_W_INT8: return plan_w<FP_W_INT8>(epi, M, N, K);
    default: return plan_w<FP_W_INT4_G128>(epi, M, N, K);
  }
}

template <int WQ, int NT, int EPI>
static cudaError_t launch_mma_t(const uint16_t* x, int M, int N, int K, const void* codes, const uint16_t* scales,
                                const uint16_t* zeros, const uint16_t* R, void* y, void* ws, size_t ws_bytes,
                                cudaStream_t s, int32_t* err) {
  const GemvPlan p = plan_t<WQ, NT, EPI>(M, N, K);
  if (p.ctas <= 0) return cudaErrorInvalidValue;
  // never launch with less workspace than this plan writes; partials are read as float4
  if (!ws || ws_bytes < p.ws || ((uintptr_t)ws & 15)) return cudaErrorInvalidValue;
  unsigned* counters = (unsigned*)ws;
  float* part = (float*)((char*)ws + counter_bytes(p.blocks));
  return launch(gemv_mma_kernel<WQ, NT, EPI>, dim3(p.ctas), dim3(kGemvWarps * 32), p.smem, s, x, M, N, K, codes,
                scales, zeros, R, y, p.total, p.S, p.W, part, counters, err);
}

template <int WQ, int EPI>
static cudaError_t launch_mma_e(const uint16_t* x, int M, int N, int K, const void* codes, const uint16_t* scales,
                                const uint16_t* zeros, const uint16_t* R, void* y, void* ws, size_t ws_bytes,
                                cudaStream_t s, int32_t* err) {
  switch (gemv_nt(M)) {
    case 1: return launch_mma_t<WQ, 1, EPI>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
    case 2: return launch_mma_t<WQ, 2, EPI>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
    case 4: return launch_mma_t<WQ, 4, EPI>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
    default: return launch_mma_t<WQ, 8, EPI>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
  }
}

template <int WQ>
static cudaError_t launch_mma(int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                              const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* y, void* ws,
                              size_t ws_bytes, cudaStream_t s, int32_t* err) {
  switch (epi) {
    case FP_EPI_STORE: return launch_mma_e<WQ, FP_EPI_STORE>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
    case FP_EPI_RESID: return launch_mma_e<WQ, FP_EPI_RESID>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
    case FP_EPI_SWIGLU: return launch_mma_e<WQ, FP_EPI_SWIGLU>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
    default: return launch_mma_e<WQ, FP_EPI_F32>(x, M, N, K, codes, scales, zeros, R, y, ws, ws_bytes, s, err);
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
  size_t w = 0;
  for (int epi : {FP_EPI_STORE, FP_EPI_RESID, FP_EPI_F32, FP_EPI_SWIGLU}) {
    if (epi == FP_EPI_SWIGLU && N % 2 != 0) continue;
    if (mma_ok(wquant, M, N, K)) w = std::max(w, plan_for(wquant, epi, M, N, K).ws);
    if (q4tc_ok(wquant, epi, M, N, K)) w = std::max(w, q4tc_ws_bytes(epi, M, N, K));
    if (btc_ok(wquant, epi, M, N, K)) w = std::max(w, btc_ws_bytes(epi, M, N, K));
  }
  return w;
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
    // int8 / int4 without room for the bf16 expansion: dequantise inside the GEMM
    if (need > 0 && (!ws || ws_bytes < need) && gemm_wq_ok(wquant, epi, M, N, K, x, codes))
      return launch_gemm_wq(wquant, epi, x, M, N, K, codes, scales, zeros, residual, y, err, s);
    if (need > 0 && (!ws || ws_bytes < need)) return cudaErrorInvalidValue;
    void* scratch = need ? (char*)ws + counter_bytes(0) : nullptr;
    return launch_gemm_tc(wquant, epi, x, M, N, K, codes, scales, zeros, residual, y, scratch,
                          need ? ws_bytes - counter_bytes(0) : 0, err, s);
  }
  // bf16 weights at 17-64 tokens: the TMA-fed tcgen05 GEMV where every SM gets
  // enough 32 KB items to hide their per-item cost (16-byte aligned x and weights)
  if (btc_ok(wquant, epi, M, N, K) && btc_preferred(epi, N, K) && ((uintptr_t)x & 15) == 0 &&
      ((uintptr_t)codes & 15) == 0)
    return launch_btc(epi, x, M, N, K, codes, residual, y, ws, ws_bytes, err, s);
  // int4 and int8 at 17-64 tokens: the tensor-core path, weights expanded into
  // TMEM (TMA needs 16-byte aligned x and codes)
  if (q4tc_ok(wquant, epi, M, N, K) && q4tc_preferred(wquant, M, K) && ((uintptr_t)x & 15) == 0 &&
      ((uintptr_t)codes & 15) == 0)
    return launch_q4tc(wquant, epi, x, M, N, K, codes, scales, zeros, residual, y, ws, ws_bytes, err, s);
  if (mma_ok(wquant, M, N, K)) {
    switch (wquant) {
      case FP_W_BF16: return launch_mma<FP_W_BF16>(epi, x, M, N, K, codes, scales, zeros, residual, y, ws, ws_bytes, s, err);
      case FP_W_INT8: return launch_mma<FP_W_INT8>(epi, x, M, N, K, codes, scales, zeros, residual, y, ws, ws_bytes, s, err);
      default: return launch_mma<FP_W_INT4_G128>(epi, x, M, N, K, codes, scales, zeros, residual, y, ws, ws_bytes, s, err);
    }
  }
  switch (wquant) {
    case FP_W_BF16: return launch_gemv<FP_W_BF16>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
    case FP_W_INT8: return launch_gemv<FP_W_INT8>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
    default: return launch_gemv<FP_W_INT4_G128>(epi, x, M, N, K, codes, scales, zeros, residual, y, s);
  }
}

}  // namespace fpk

namespace fpk {

// ---- GPTQ4 (int4 over an act order)
// Decode (M <= 64): the workspace holds the int4 linear's own workspace
// (ticket area first, kept at offset 0 whatever the shape) and then x in act
// order, xp[m][j] = x[m][perm[j]]; the stored matrix is a plain int4 g128
// matrix of the act-order channels, so y = xp W_stored^T.  Prefill: the
// bf16 expansion puts each weight back in channel order (inv, the inverse
// act order; computed into the workspace when the caller passes none) and
// the GEMM multiplies x as it is.
static size_t align256(size_t b) { return (b + 255) / 256 * 256; }

static size_t gptq4_xp_offset(int M, int N, int K) {
  return align256(std::max(linear_ws_bytes(FP_W_INT4_G128, M, N, K), counter_bytes(0)));
}

size_t linear_gptq4_ws_bytes(int M, int N, int K, bool with_inv) {
  if (M <= 0 || N <= 0 || K <= 0) return 0;
  if (M > 64) return align256(std::max(linear_ws_bytes(FP_W_INT4_G128, M, N, K), counter_bytes(0))) +
                     (with_inv ? align256((size_t)K * 4) : 0);
  return gptq4_xp_offset(M, N, K) + align256((size_t)M * K * 2);
}

size_t linear_gptq4_ws_bytes_upto(int max_m, int N, int K, bool with_inv) {
  size_t w = 0;
  for (int m = 1; m <= std::min(max_m, 64); ++m) w = std::max(w, linear_gptq4_ws_bytes(m, N, K, with_inv));
  if (max_m > 64) w = std::max(w, linear_gptq4_ws_bytes(max_m, N, K, with_inv));
  return w;
}

cudaError_t launch_linear_gptq4(int epi, const uint16_t* x, int M, int N, int K, const int32_t* perm,
                                const int32_t* inv, const void* codes, const uint16_t* scales,
                                const uint16_t* zeros, const uint16_t* residual, void* y, void* ws, size_t ws_bytes,
                                cudaStream_t s, int32_t* err) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  if (!ws || ws_bytes < linear_gptq4_ws_bytes(M, N, K, inv == nullptr)) return cudaErrorInvalidValue;
  if (M > 64) {
    if (!gemm_tc_ok(M, N, K)) return cudaErrorInvalidValue;
    const size_t lin = align256(std::max(linear_ws_bytes(FP_W_INT4_G128, M, N, K), counter_bytes(0)));
    if (!inv) {
      int32_t* tmp = (int32_t*)((char*)ws + lin);
      FP_CUDA_TRY(launch_invert_perm(perm, K, tmp, err, s));
      inv = tmp;
    }
    return launch_gemm_tc(FP_W_GPTQ4, epi, x, M, N, K, codes, scales, zeros, residual, y,
                          (char*)ws + counter_bytes(0), lin - counter_bytes(0), err, s, inv);
  }
  uint16_t* xp = (uint16_t*)((char*)ws + gptq4_xp_offset(M, N, K));
  FP_CUDA_TRY(launch_gather_cols(x, M, K, perm, xp, err, s));
  return launch_linear(FP_W_INT4_G128, epi, xp, M, N, K, codes, scales, zeros, residual, y, ws,
                       gptq4_xp_offset(M, N, K), s, err);
}

}  // namespace fpk
