// Prefill weight-only linear on the 5th-generation tensor cores.
//
// y[M][N] = x[M][K] W[N][K]^T for M > 64 (prefill), the dense contraction of
// the block's linear layers.  One persistent CTA per SM walks 128 x 256
// output tiles, each over the whole K:
//   warp 0      TMA producer: x tile [128][64] and W tile [256][64] (bf16,
//               128-byte swizzled, K-major) into a 4-stage shared ring,
//               completion counted in bytes on mbarrier full[s];
//   warp 1      allocates 512 TMEM columns (two fp32 accumulators) and, from
//               one thread, issues tcgen05.mma (M 128, N 256, K 16);
//               tcgen05.commit frees each stage (empty[s]) and signals a full
//               accumulator (tfull[b]);
//   warps 2-5   epilogue: tcgen05.ld of the accumulator (one TMEM lane per
//               output row), per-column int8 scale, residual add / SwiGLU /
//               fp32 store; then the buffer goes back to the MMA thread
//               (tempty[b]) while the next tile accumulates in the other.
// Quantised weights are first expanded to bf16 into a scratch matrix by
// dequant_kernel (int8: the code itself, exact, with its row scale applied
// in the epilogue; int4: bf16((q - z) * s)).
//
// Every mbarrier wait is bounded: past the limit the thread records an error
// in the error word, the CTA stops issuing work and falls through to the TMEM
// release, so a fault in the pipeline surfaces as a status, not a hang.
#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

// Rounds after which the MMA thread's wait for a stage gives up: kTcSpinLimit,
// unless a test lowers it through fp_debug_set_wait_limit to run the failure
// path (every other wait keeps kTcSpinLimit, so copies and MMAs in flight are
// still drained before the CTA leaves).
static __device__ long long g_stage_wait_limit = fpk::kTcSpinLimit;

namespace fpk {

constexpr int kTcBM = 128, kTcBN = 256, kTcBK = 64, kTcStages = 4;
constexpr int kTcThreads = 192;
constexpr uint32_t kTcStageBytes = (kTcBM + kTcBN) * kTcBK * 2;  // 48 KiB
constexpr uint32_t kTcTmemCols = 512;  // two 256-column fp32 accumulators

// ------------------------------------------------------------------ kernel
// Persistent: CTA c takes output tiles c, c + gridDim.x, ... in grouped
// order (16 M tiles share each sweep over the N tiles, so a wave's x rows
// and weight columns stay in L2).  The shared ring runs across tiles, and
// the fp32 accumulator is double-buffered in TMEM (2 x 256 columns): the MMA
// thread fills one buffer while the epilogue warps drain the other.
// SCALE: multiply output column n by bf16 scales[n] (int8 weights; SwiGLU:
// the up column by scales[up_off + n]).  Output (and residual) rows are ldy
// elements apart, so a launch can fill a band of columns of a wider output.
template <int EPI, bool SCALE>
__global__ void __launch_bounds__(kTcThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap map_x, const __grid_constant__ CUtensorMap map_w, int M, int N,
                   int K, const uint16_t* __restrict__ scales, long long up_off, const uint16_t* R, void* Y,
                   int ldy, int32_t* err) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t full[kTcStages], empty[kTcStages], tfull[2], tempty[2], mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_word;
  volatile int* abort_flag = &abort_word;  // set by a role that gave up waiting
  // stage buffers must be 1024-byte aligned for the 128-byte swizzle
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  const int Nout = NR == 2 ? N / 2 : N;
  constexpr int BNout = kTcBN / NR;
  const int tiles_m = (M + kTcBM - 1) / kTcBM, tiles_n = (Nout + BNout - 1) / BNout;
  const int ntiles = tiles_m * tiles_n;
  const int kblocks = (K + kTcBK - 1) / kTcBK;
  auto tile_origin = [&](int t, int& m0, int& n0) {
    constexpr int GM = 16;
    const int span = GM * tiles_n;
    const int first = (t / span) * GM;
    const int gs = min(GM, tiles_m - first);
    const int r = t % span;
    m0 = (first + r % gs) * kTcBM;
    n0 = (r / gs) * BNout;
  };

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);   // tcgen05.commit of the tile's last MMAs
      mbar_init(&tempty[b], 4);  // one arrival per epilogue warp
    }
    mbar_init(&mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                 "r"(kTcTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  pdl_wait();

  if (warp == 0) {
    // ---------------- TMA producer
    if (lane == 0) {
      int it = 0;  // k-blocks issued, across tiles
      for (int t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x) {
        int m0, n0;
        tile_origin(t, m0, n0);
        for (int kb = 0; kb < kblocks; ++kb, ++it) {
          const int s = it % kTcStages;
          if (!mbar_wait(&empty[s], ((it / kTcStages) & 1) ^ 1) || *abort_flag) {
            *abort_flag = 1;
            if (err) atomicExch(err, 2);
            break;
          }
          uint8_t* a = smem + s * kTcStageBytes;
          uint8_t* b = a + kTcBM * kTcBK * 2;
          mbar_expect_tx(&full[s], kTcStageBytes);
          tma_load_2d(a, &map_x, kb * kTcBK, m0, &full[s]);
          if (NR == 1) {
            tma_load_2d(b, &map_w, kb * kTcBK, n0, &full[s]);
          } else {
            tma_load_2d(b, &map_w, kb * kTcBK, n0, &full[s]);                              // gate rows
            tma_load_2d(b + 128 * kTcBK * 2, &map_w, kb * kTcBK, Nout + n0, &full[s]);  // up rows
          }
        }
      }
      // copies still in flight land before the CTA leaves (their stages are its shared memory)
      for (int j = max(0, it - kTcStages); j < it; ++j) mbar_wait(&full[j % kTcStages], (j / kTcStages) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc(kTcBM, kTcBN);
      const long long stage_limit = g_stage_wait_limit;
      int it = 0, lt = 0;
      for (int t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x, ++lt) {
        const int acc = lt & 1;
        // the epilogue has drained this accumulator (local tile lt - 2)
        if (!mbar_wait(&tempty[acc], ((lt >> 1) & 1) ^ 1) || *abort_flag) {
          *abort_flag = 1;
          if (err) atomicExch(err, 2);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)acc * kTcBN;
        bool ok = true;
        for (int kb = 0; kb < kblocks; ++kb, ++it) {
          const int s = it % kTcStages;
          if (!mbar_wait_n(&full[s], (it / kTcStages) & 1, stage_limit) || *abort_flag) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a = smem_u32(smem + s * kTcStageBytes);
          const uint32_t b = a + kTcBM * kTcBK * 2;
#pragma unroll
          for (int kk = 0; kk < kTcBK / 16; ++kk)
            tc_mma(d, sdesc(a + kk * 32), sdesc(b + kk * 32), idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          tc_commit(&empty[s]);  // stage s is free once these MMAs have read it
        }
        if (!ok) {
          *abort_flag = 1;
          if (err) atomicExch(err, 2);
          break;
        }
        tc_commit(&tfull[acc]);  // the tile's accumulator is complete
      }
      // every MMA issued has completed before TMEM is released
      tc_commit(&mma_done);
      mbar_wait(&mma_done, 0);
    }
  } else {
    // ---------------- epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31
    const int q = warp & 3;
    int lt = 0;
    for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++lt) {
      const int acc = lt & 1;
      int m0, n0;
      tile_origin(t, m0, n0);
      const bool ok = mbar_wait(&tfull[acc], (lt >> 1) & 1);
      if (!ok || *abort_flag) {
        if (!ok && err) atomicExch(err, 2);
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const int row = m0 + q * 32 + lane;
      const uint32_t tl = tmem + (uint32_t)acc * kTcBN + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
      for (int c0 = 0; c0 < BNout; c0 += 32) {
        float v[32], u[32];
        tc_ld32(tl + c0, v);
        if (NR == 2) tc_ld32(tl + 128 + c0, u);
        if (row >= M) continue;
        const int n = n0 + c0;
        if (n >= Nout) continue;
        const int cnt = min(32, Nout - n);
        if constexpr (SCALE) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            if (i < cnt) {
              v[i] *= bf2f(scales[n + i]);
              if (NR == 2) u[i] *= bf2f(scales[up_off + n + i]);
            }
          }
        }
        const long long o = (long long)row * ldy + n;
        if constexpr (EPI == FP_EPI_F32) {
          float* y = (float*)Y + o;
          if (cnt == 32 && (o & 3) == 0) {
#pragma unroll
            for (int i = 0; i < 32; i += 4) *reinterpret_cast<float4*>(y + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
          } else {
            for (int i = 0; i < cnt; ++i) y[i] = v[i];
          }
        } else {
          uint16_t* y = (uint16_t*)Y + o;
          float r[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            if constexpr (EPI == FP_EPI_SWIGLU) r[i] = silu(v[i]) * u[i];
            else r[i] = v[i];
          }
          if constexpr (EPI == FP_EPI_RESID) {
            const uint16_t* rr = R + o;
            for (int i = 0; i < cnt; ++i) r[i] += bf2f(rr[i]);
          }
          if (cnt == 32 && (o & 7) == 0) {
#pragma unroll
            for (int i = 0; i < 32; i += 8)
              *reinterpret_cast<uint4*>(y + i) = make_uint4(pack_bf2(r[i], r[i + 1]), pack_bf2(r[i + 2], r[i + 3]),
                                                            pack_bf2(r[i + 4], r[i + 5]), pack_bf2(r[i + 6], r[i + 7]));
          } else {
            for (int i = 0; i < cnt; ++i) y[i] = f2bf(r[i]);
          }
        }
      }
      // this warp's reads of the accumulator are done: hand the buffer back to the MMA thread
      tc_fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&tempty[acc])) : "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcTmemCols) : "memory");
  }
}

// ------------------------------------------------------------------ dequant to bf16
// int8: w = q (exact; the row scale is applied by the GEMM epilogue).
// int4: w = bf16((q - z) * s), 8 elements (one packed word) per thread.
// GPTQ4: the same expansion back into channel order: output channel k is
// act-order column j = inv[k] (inv the inverse of the act order), with the
// scale and zero of group j / 128; 8 consecutive channels per thread.
__global__ void dequant_kernel(int wquant, const void* __restrict__ codes, const uint16_t* __restrict__ scales,
                               const uint16_t* __restrict__ zeros, int N, int K, uint16_t* __restrict__ out,
                               const int32_t* __restrict__ inv) {
  pdl_trigger();
  pdl_wait();
  const long long words = (long long)N * K / 8;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < words; i += (long long)gridDim.x * blockDim.x) {
    const long long e0 = i * 8;
    const long long row = e0 / K;
    const int k0 = (int)(e0 % K);
    float f[8];
    if (wquant == FP_W_GPTQ4) {
      const uint32_t* cw = (const uint32_t*)codes + row * (K / 8);
      const long long g0 = row * (K / 128);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int a = min(max(inv[k0 + j], 0), K - 1);  // the inverse comes from the act order, in range
        const int e = a & 7, nib = (e >> 1) + 4 * (e & 1);  // element e of a word sits in this nibble
        const float q = (float)((cw[a >> 3] >> (4 * nib)) & 0xF);
        f[j] = (q - bf2f(zeros[g0 + (a >> 7)])) * bf2f(scales[g0 + (a >> 7)]);
      }
    } else if (wquant == FP_W_INT8) {
      const uint2 c = *reinterpret_cast<const uint2*>((const int8_t*)codes + e0);
      const uint32_t w[2] = {c.x, c.y};
#pragma unroll
      for (int j = 0; j < 8; ++j) f[j] = (float)(int8_t)((w[j >> 2] >> (8 * (j & 3))) & 0xFF);
    } else {
      const uint32_t w = *reinterpret_cast<const uint32_t*>((const uint8_t*)codes + e0 / 2);
      const long long gi = row * (K / 128) + k0 / 128;
      const float s = bf2f(scales[gi]), z = bf2f(zeros[gi]);
      // nibbles i and i + 4 hold elements 2i and 2i + 1
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        f[2 * j] = ((float)((w >> (4 * j)) & 0xF) - z) * s;
        f[2 * j + 1] = ((float)((w >> (4 * j + 16)) & 0xF) - z) * s;
      }
    }
    *reinterpret_cast<uint4*>(out + e0) =
        make_uint4(pack_bf2(f[0], f[1]), pack_bf2(f[2], f[3]), pack_bf2(f[4], f[5]), pack_bf2(f[6], f[7]));
  }
}

// ------------------------------------------------------------------ host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &p, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeTiledFn)p;
  }
  return fn;
}

bool make_tensor_map(CUtensorMap* map, const void* base, long long rows, long long cols, int elem_bytes,
                     int box_rows, int box_cols, int swizzle_bytes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || (elem_bytes != 1 && elem_bytes != 2 && elem_bytes != 4) || (swizzle_bytes != 64 && swizzle_bytes != 128))
    return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * elem_bytes};
  cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  const CUtensorMapDataType dt = elem_bytes == 4   ? CU_TENSOR_MAP_DATA_TYPE_UINT32
                                 : elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16
                                                   : CU_TENSOR_MAP_DATA_TYPE_UINT8;
  return fn(map, dt, 2,
            const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            swizzle_bytes == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tensor_maps_available() { return encode_fn() != nullptr; }

// bf16 [rows][cols] row-major, box [box_rows][64] with 128-byte swizzle.
static bool make_map(CUtensorMap* map, const void* base, long long rows, long long cols, int box_rows) {
  return make_tensor_map(map, base, rows, cols, 2, box_rows, kTcBK, 128);
}

// Quantised weights are expanded to bf16 band by band of output columns, so
// the scratch holds at most kTcScratchBytes (or one band of 256 columns).
constexpr size_t kTcScratchBytes = 128u << 20;

// Output columns per band: a multiple of the tile's (256, SwiGLU 128), all of them if they fit.
static int band_cols(int epi, int N, int K) {
  const int nr = epi == FP_EPI_SWIGLU ? 2 : 1;
  const int nout = nr == 2 ? N / 2 : N;
  const int unit = kTcBN / nr;
  const long long fit = (long long)(kTcScratchBytes / ((size_t)nr * K * 2)) / unit * unit;
  return (int)std::min<long long>(nout, std::max<long long>(unit, fit));
}

size_t gemm_tc_ws_bytes(int wquant, int N, int K) {
  if (wquant == FP_W_BF16) return 0;
  // the largest band over the epilogues (a SwiGLU band holds its gate and its up rows)
  const size_t plain = (size_t)band_cols(FP_EPI_STORE, N, K) * K * 2;
  const size_t swiglu = N % 2 == 0 ? (size_t)2 * band_cols(FP_EPI_SWIGLU, N, K) * K * 2 : 0;
  return std::max(plain, swiglu);
}

bool gemm_tc_ok(int M, int N, int K) { return M > 64 && K % 8 == 0 && N >= 1 && encode_fn() != nullptr; }

template <int EPI, bool SCALE>
static cudaError_t launch_tc_t(const CUtensorMap& mx, const CUtensorMap& mw, int M, int N, int K,
                               const uint16_t* scales, long long up_off, const uint16_t* R, void* Y, int ldy,
                               int32_t* err, cudaStream_t s) {
  auto kern = gemm_tc_kernel<EPI, SCALE>;
  const size_t smem = (size_t)kTcStages * kTcStageBytes + 1024;
  static std::atomic<unsigned long long> attr{0};
  FP_CUDA_TRY(smem_limit_once(kern, (int)smem, &attr));
  const int Nout = EPI == FP_EPI_SWIGLU ? N / 2 : N;
  const int bn = kTcBN / (EPI == FP_EPI_SWIGLU ? 2 : 1);
  const long long tiles = (long long)((Nout + bn - 1) / bn) * ((M + kTcBM - 1) / kTcBM);
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        sms <= 0)
      sms = 152;
  }
  // persistent: one CTA per SM (its shared ring and 512 TMEM columns fill the SM)
  const dim3 grid((unsigned)std::min<long long>(tiles, sms));
  return launch(kern, grid, dim3(kTcThreads), smem, s, mx, mw, M, N, K, scales, up_off, R, Y, ldy, err);
}

template <int EPI>
static cudaError_t launch_tc_e(bool sc, const CUtensorMap& mx, const CUtensorMap& mw, int M, int N, int K,
                               const uint16_t* scales, long long up_off, const uint16_t* R, void* Y, int ldy,
                               int32_t* err, cudaStream_t s) {
  return sc ? launch_tc_t<EPI, true>(mx, mw, M, N, K, scales, up_off, R, Y, ldy, err, s)
            : launch_tc_t<EPI, false>(mx, mw, M, N, K, scales, up_off, R, Y, ldy, err, s);
}

static cudaError_t launch_tc_any(int epi, bool sc, const CUtensorMap& mx, const CUtensorMap& mw, int M, int N, int K,
                                 const uint16_t* scales, long long up_off, const uint16_t* R, void* Y, int ldy,
                                 int32_t* err, cudaStream_t s) {
  switch (epi) {
    case FP_EPI_STORE: return launch_tc_e<FP_EPI_STORE>(sc, mx, mw, M, N, K, scales, up_off, R, Y, ldy, err, s);
    case FP_EPI_RESID: return launch_tc_e<FP_EPI_RESID>(sc, mx, mw, M, N, K, scales, up_off, R, Y, ldy, err, s);
    case FP_EPI_SWIGLU: return launch_tc_e<FP_EPI_SWIGLU>(sc, mx, mw, M, N, K, scales, up_off, R, Y, ldy, err, s);
    default: return launch_tc_e<FP_EPI_F32>(sc, mx, mw, M, N, K, scales, up_off, R, Y, ldy, err, s);
  }
}

// Expand rows [r0, r0 + rows) of a quantised matrix into out [rows][K] bf16.
static cudaError_t dequant_rows(int wquant, const void* codes, const uint16_t* scales, const uint16_t* zeros, long long r0,
                                int rows, int K, uint16_t* out, const int32_t* inv, cudaStream_t s) {
  const bool grouped = wquant == FP_W_INT4_G128 || wquant == FP_W_GPTQ4;
  const uint8_t* c = (const uint8_t*)codes + (wquant == FP_W_INT8 ? r0 * K : r0 * (K / 2));
  const uint16_t* sc = grouped ? scales + r0 * (K / 128) : scales;
  const uint16_t* ze = grouped ? zeros + r0 * (K / 128) : zeros;
  const long long words = (long long)rows * K / 8;
  const int blocks = (int)std::min<long long>((words + 255) / 256, 152 * 16);
  return launch(dequant_kernel, dim3(blocks), dim3(256), 0, s, wquant, (const void*)c, sc, ze, rows, K, out, inv);
}

cudaError_t launch_gemm_tc(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                           const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                           void* ws, size_t ws_bytes, int32_t* err, cudaStream_t s, const int32_t* inv) {
  const int nr = epi == FP_EPI_SWIGLU ? 2 : 1;
  const int Nout = nr == 2 ? N / 2 : N;
  const int wbox = epi == FP_EPI_SWIGLU ? 128 : 256;
  const bool sc = wquant == FP_W_INT8;
  CUtensorMap mx, mw;
  if (!make_map(&mx, x, M, K, kTcBM)) return cudaErrorInvalidValue;
  if (wquant == FP_W_BF16) {
    if (!make_map(&mw, codes, N, K, wbox)) return cudaErrorInvalidValue;
    return launch_tc_any(epi, sc, mx, mw, M, N, K, scales, Nout, residual, y, Nout, err, s);
  }
  if (!ws || ws_bytes < gemm_tc_ws_bytes(wquant, N, K)) return cudaErrorInvalidValue;
  // band by band of output columns: expand the band's rows (SwiGLU: its gate
  // rows, then its up rows) into the scratch, then multiply
  uint16_t* w = (uint16_t*)ws;
  const int band = band_cols(epi, N, K);
  for (int c0 = 0; c0 < Nout; c0 += band) {
    const int cols = std::min(band, Nout - c0);
    FP_CUDA_TRY(dequant_rows(wquant, codes, scales, zeros, c0, cols, K, w, inv, s));
    if (nr == 2)
      FP_CUDA_TRY(dequant_rows(wquant, codes, scales, zeros, (long long)Nout + c0, cols, K, w + (size_t)cols * K, inv, s));
    if (!make_map(&mw, w, (long long)nr * cols, K, wbox)) return cudaErrorInvalidValue;
    const uint16_t* r = residual ? residual + c0 : nullptr;
    void* yb = epi == FP_EPI_F32 ? (void*)((float*)y + c0) : (void*)((uint16_t*)y + c0);
    FP_CUDA_TRY(launch_tc_any(epi, sc, mx, mw, M, nr * cols, K, sc ? scales + c0 : scales, Nout, r, yb, Nout, err, s));
  }
  return cudaSuccess;
}

}  // namespace fpk

extern "C" int fp_debug_set_wait_limit(long long rounds) {
  const long long v = rounds < 0 ? fpk::kTcSpinLimit : std::min(rounds, fpk::kTcSpinLimit);
  return cudaMemcpyToSymbol(g_stage_wait_limit, &v, sizeof v) == cudaSuccess ? FP_OK : FP_ERR_CUDA;
}
