// Decode linear for bf16 weights at 17-64 tokens on the tcgen05 tensor cores.
//
// y[m][n] = sum_k x[m][k] W[n][k]: the LM head of a decode step (fp32 out)
// and the block linears of the bf16-weight configurations, while the batch
// is large enough that the mma.sync GEMV's per-token work (one MMA per 8
// tokens per weight fragment, x fragments from shared memory) bounds it.  No
// conversion is needed, so TMA streams the weights straight into the MMA:
//   warp 0      TMA producer: per item the weight tiles [128][64] bf16 (two
//               consecutive k-blocks of one row tile, or SwiGLU one k-block
//               of the gate and of the up tile) and the matching x tiles
//               [MT][64], 128-byte swizzled and K-major, into a ring of 4-6
//               stages (full[s], bytes counted);
//   warp 1      allocates TMEM and issues tcgen05.mma (M 128 weight rows, N =
//               tokens rounded up to 32 or 64, K 16) into one of two
//               accumulator buffers; tcgen05.commit frees the stage and, at
//               the end of a row tile's k range, hands the buffer to the
//               epilogue (tfull / tempty);
//   warps 2-5   epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31, one
//               weight row (output column) per thread over all tokens.
// The (row tile, k-block) items are split into equal contiguous ranges, one
// per CTA (stream-K, as the other decode linears): a CTA whose range covers a
// whole row tile runs the epilogue itself; otherwise each epilogue warp
// writes fp32 partials of its 32 rows, and the last CTA to finish that slice
// (a ticket per slice) sums them in CTA order and runs the epilogue --
// residual add, SwiGLU, bf16 or fp32 store.  Nothing spins on another CTA.
//
// Every mbarrier wait is bounded; past the limit the thread records error 2
// in the error word and the CTA stops, after its copies and MMAs in flight
// have completed and before TMEM is released.
#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace fpk {

constexpr int kBtRows = 128, kBtBK = 64;
constexpr int kBtThreads = 6 * 32;  // TMA, MMA, four epilogue warps

// An item is 32 KB of weights: without SwiGLU two 64-k sub-blocks of one
// row tile (KBI = 2), with SwiGLU one sub-block of the gate and of the up
// tile; half-size items measured slower (their per-item overheads dominate).
template <int MT, int NR>
struct BtGeom {
  static constexpr int KBI = NR == 1 ? 2 : 1;                     // 64-k sub-blocks per item
  static constexpr int kTile = kBtRows * kBtBK * 2;                // one [128][64] bf16 box
  static constexpr int kABytes = NR * KBI * kTile;                 // weight boxes of an item
  static constexpr int kXBox = MT * kBtBK * 2;                     // one [MT][64] x box
  static constexpr int kXBytes = KBI * kXBox;
  static constexpr int kStage = kABytes + kXBytes;
  static constexpr int kStages = std::min(8, (int)(220 * 1024 / kStage));  // ring depth within shared memory
  static constexpr int kSmem = kStages * kStage + 1024;
  static constexpr int kDCols = NR * MT;  // one accumulator buffer
  static constexpr uint32_t kTmemCols = 2 * kDCols < 32 ? 32u : (uint32_t)(2 * kDCols);
  static_assert(kStage % 1024 == 0 && kXBox % 1024 == 0, "stages stay 1024-byte aligned");
  static_assert(kSmem <= 227 * 1024, "shared memory");
};

FP_DEV long long bt_cta_of(long long i, long long C, long long total) { return ((i + 1) * C - 1) / total; }

template <int MT, int EPI>
__global__ void __launch_bounds__(kBtThreads, 1)
    gemv_btc_kernel(const __grid_constant__ CUtensorMap map_w, const __grid_constant__ CUtensorMap map_x, int M,
                    int N, const uint16_t* R, void* Y, long long total, int S, float* __restrict__ ws,
                    unsigned* __restrict__ counters, int32_t* err) {
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  using G = BtGeom<MT, NR>;
  constexpr int ST = G::kStages;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t full[ST], empty[ST], tfull[2], tempty[2], mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_word;
  volatile int* abort_flag = &abort_word;
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Nout = NR == 2 ? N / 2 : N;
  const long long C = gridDim.x, c = blockIdx.x;
  const long long begin = c * total / C, end = (c + 1) * total / C;
  const int L = (int)(end - begin);
  auto fail = [&]() {
    *abort_flag = 1;
    if (err) atomicExch(err, 2);
  };

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < ST; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);
    }
    mbar_init(&mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                 "r"(G::kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 0) {
    // ---------------- TMA producer: the weights are constant, so the ring fills
    // before the previous kernel has finished; x waits for it
    if (lane == 0) {
      int issued = 0;
      bool waited = false;
      for (int q = 0; q < L; ++q) {
        const long long p = begin + q;
        const int b = (int)(p / S), kb = (int)(p % S);
        const int s = q % ST;
        if (q >= ST && (!mbar_wait(&empty[s], ((q / ST) & 1) ^ 1) || *abort_flag)) {
          fail();
          break;
        }
        uint8_t* a = smem + s * G::kStage;
        mbar_expect_tx(&full[s], G::kStage);
#pragma unroll
        for (int j = 0; j < G::KBI; ++j) {
          const int k0 = (kb * G::KBI + j) * kBtBK;  // past K the boxes read zeros
          tma_load_2d(a + j * G::kTile, &map_w, k0, b * kBtRows, &full[s]);
          if (NR == 2) tma_load_2d(a + G::kTile, &map_w, k0, Nout + b * kBtRows, &full[s]);
        }
        if (!waited) {
          pdl_wait();  // x is the previous kernel's output
          waited = true;
        }
#pragma unroll
        for (int j = 0; j < G::KBI; ++j)
          tma_load_2d(a + G::kABytes + j * G::kXBox, &map_x, (kb * G::KBI + j) * kBtBK, 0, &full[s]);
        issued = q + 1;
      }
      if (!waited) pdl_wait();
      // copies still in flight land before the CTA leaves (their stages are its shared memory)
      for (int j = max(0, issued - ST); j < issued; ++j) mbar_wait(&full[j % ST], (j / ST) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc(kBtRows, MT);
      bool ok = true;
      int seg = 0;
      for (int q = 0; q < L && ok; ++q) {
        const long long p = begin + q;
        const int kb = (int)(p % S);
        const bool first = q == 0 || kb == 0, last = kb == S - 1 || q == L - 1;
        const int buf = seg & 1;
        if (first && seg >= 2) ok = mbar_wait(&tempty[buf], ((seg >> 1) & 1) ^ 1);  // the epilogue drained it
        const int s = q % ST;
        ok = ok && mbar_wait(&full[s], (q / ST) & 1) && !*abort_flag;
        if (!ok) break;
        tc_fence_after();
        const uint32_t a = smem_u32(smem + s * G::kStage), xb = a + G::kABytes;
#pragma unroll
        for (int r = 0; r < NR; ++r)
#pragma unroll
          for (int j = 0; j < G::KBI; ++j)
#pragma unroll
            for (int kk = 0; kk < kBtBK / 16; ++kk)
              tc_mma(tmem + buf * G::kDCols + r * MT, sdesc(a + (r + j) * G::kTile + kk * 32),
                     sdesc(xb + j * G::kXBox + kk * 32), idesc, (first && j == 0 && kk == 0) ? 0u : 1u);
        tc_commit(&empty[s]);  // the stage is free once these MMAs have read it
        if (last) {
          tc_commit(&tfull[buf]);
          ++seg;
        }
      }
      if (!ok) fail();
      tc_commit(&mma_done);  // every MMA issued has completed before TMEM is released
      mbar_wait(&mma_done, 0);
    }
  } else {
    // ---------------- epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31
    const int qd = warp & 3, ew = warp - 2, lr = qd * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(qd * 32) << 16);
    const int b0 = (int)(begin / S), b1 = L > 0 ? (int)((end - 1) / S) : b0 - 1;
    pdl_wait();  // the residual and the output follow the stream's order
    int seg = 0;
    for (int b = b0; b <= b1; ++b, ++seg) {
      const int buf = seg & 1;
      const bool got = __all_sync(0xffffffffu, mbar_wait(&tfull[buf], (seg >> 1) & 1));
      if (!got || __any_sync(0xffffffffu, *abort_flag != 0)) {
        if (lane == 0) fail();
        break;
      }
      tc_fence_after();
      uint32_t dv[NR][MT];
#pragma unroll
      for (int r = 0; r < NR; ++r) tc_ld<MT>(lane_base + buf * G::kDCols + r * MT, dv[r]);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[buf]);

      const int row = b * kBtRows + lr;
      // r: the residual R[m][row], read before any store (R may be Y itself)
      auto resid = [&](int m) {
        return (EPI == FP_EPI_RESID && m < M && row < Nout) ? bf2f(R[(long long)m * Nout + row]) : 0.f;
      };
      auto finish = [&](int m, float v, float u, float r) {
        const long long o = (long long)m * Nout + row;
        if constexpr (EPI == FP_EPI_STORE) ((uint16_t*)Y)[o] = f2bf(v);
        else if constexpr (EPI == FP_EPI_RESID) ((uint16_t*)Y)[o] = f2bf(r + v);
        else if constexpr (EPI == FP_EPI_SWIGLU) ((uint16_t*)Y)[o] = f2bf(silu(v) * u);
        else ((float*)Y)[o] = v;
      };
      const long long c0 = bt_cta_of((long long)b * S, C, total);
      const long long c1 = bt_cta_of((long long)(b + 1) * S - 1, C, total);
      if (c0 == c1) {
#pragma unroll
        for (int i0 = 0; i0 < MT; i0 += 8) {
          float rv[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) rv[i] = resid(i0 + i);
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (i0 + i < M && row < Nout)
              finish(i0 + i, __uint_as_float(dv[0][i0 + i]), __uint_as_float(dv[NR - 1][i0 + i]), rv[i]);
        }
        continue;
      }
      // partial slot b + c: distinct for every (row tile, CTA) pair that meets
      const size_t slot = (size_t)M * NR * kBtRows;
      float* part = ws + (size_t)(b + c) * slot;
#pragma unroll
      for (int i = 0; i < MT; ++i)
        if (i < M)
#pragma unroll
          for (int r = 0; r < NR; ++r) part[((size_t)i * NR + r) * kBtRows + lr] = __uint_as_float(dv[r][i]);
      __threadfence();
      __syncwarp();
      unsigned t = 0;
      if (lane == 0) t = atomicAdd(&counters[b * 4 + ew], 1u);
      t = __shfl_sync(0xffffffffu, t, 0);
      if (t != (unsigned)(c1 - c0)) continue;
      __threadfence();
      // the sum over the CTAs in CTA order (deterministic), eight tokens' loads
      // in flight per CTA rather than one
      const int cnt = (int)(c1 - c0) + 1;
      const float* p0 = ws + (size_t)(b + c0) * slot + lr;
#pragma unroll
      for (int i0 = 0; i0 < MT; i0 += 8) {
        if (i0 >= M) break;
        float v[8], u[8], rv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = u[i] = 0.f, rv[i] = resid(i0 + i);
        for (int cc = 0; cc < cnt; ++cc) {
          const float* pc = p0 + (size_t)cc * slot;
          float t[8], t2[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const bool in = i0 + i < M;
            t[i] = in ? __ldcg(pc + (size_t)(i0 + i) * NR * kBtRows) : 0.f;
            t2[i] = (NR == 2 && in) ? __ldcg(pc + (size_t)(i0 + i) * NR * kBtRows + kBtRows) : 0.f;
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) v[i] += t[i], u[i] += t2[i];
        }
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if (i0 + i < M && row < Nout) finish(i0 + i, v[i], u[i], rv[i]);
      }
      if (lane == 0) counters[b * 4 + ew] = 0u;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(G::kTmemCols) : "memory");
  }
}

// ---------------------------------------------------------------- host side
static int bt_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        n <= 0)
      n = 152;
  }
  return n;
}

bool btc_ok(int wquant, int epi, int M, int N, int K) {
  if (wquant != FP_W_BF16 || M < 17 || M > 64 || N < 1 || K < kBtBK || K % 8 != 0) return false;
  if (epi == FP_EPI_SWIGLU && N % 2 != 0) return false;
  const long long nout = epi == FP_EPI_SWIGLU ? N / 2 : N;
  const long long blocks = (nout + kBtRows - 1) / kBtRows;
  return blocks * 4 <= kLinTicketSlots && tensor_maps_available();
}

// Items per SM of a launch; below about 48 the mma.sync GEMV is faster
// (measured: 70B-shaped QKV at 32 tokens, 34 items per SM, 60 against 48 us;
// the LM head, 105 items per SM, 117 against 134 us).
bool btc_preferred(int epi, int N, int K) {
  const int nr = epi == FP_EPI_SWIGLU ? 2 : 1;
  const long long nout = nr == 2 ? N / 2 : N;
  const long long blocks = (nout + kBtRows - 1) / kBtRows;
  const int kbi = nr == 1 ? 2 : 1;
  const long long items = blocks * ((K + kbi * kBtBK - 1) / (kbi * kBtBK));
  return items >= 48LL * bt_sms();
}

size_t btc_ws_bytes(int epi, int M, int N, int K) {
  const int nr = epi == FP_EPI_SWIGLU ? 2 : 1;
  const long long nout = nr == 2 ? N / 2 : N;
  const long long blocks = (nout + kBtRows - 1) / kBtRows;
  const int kbi = nr == 1 ? 2 : 1;
  const long long kblocks = (K + kbi * kBtBK - 1) / (kbi * kBtBK);
  const long long ctas = std::min<long long>(blocks * kblocks, bt_sms());
  return (size_t)kLinTicketSlots * 4 + (size_t)(blocks + ctas) * M * nr * kBtRows * 4;
}

template <int MT, int EPI>
static cudaError_t launch_bt_t(const CUtensorMap& mw, const CUtensorMap& mx, int M, int N, int K, const uint16_t* R,
                               void* Y, void* ws, int32_t* err, cudaStream_t s) {
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  auto kern = gemv_btc_kernel<MT, EPI>;
  const int smem = BtGeom<MT, NR>::kSmem;
  static std::atomic<unsigned long long> attr{0};
  FP_CUDA_TRY(smem_limit_once(kern, smem, &attr));
  const int nout = NR == 2 ? N / 2 : N;
  const long long blocks = (nout + kBtRows - 1) / kBtRows;
  constexpr int KI = BtGeom<MT, NR>::KBI * kBtBK;  // k per item
  const int S = (K + KI - 1) / KI;
  const long long total = blocks * S;
  const int ctas = (int)std::min<long long>(total, bt_sms());
  unsigned* counters = (unsigned*)ws;
  float* part = (float*)((char*)ws + (size_t)kLinTicketSlots * 4);
  return launch(kern, dim3(ctas), dim3(kBtThreads), (size_t)smem, s, mw, mx, M, N, R, Y, total, S, part, counters,
                err);
}

template <int MT>
static cudaError_t launch_bt_m(int epi, const CUtensorMap& mw, const CUtensorMap& mx, int M, int N, int K,
                               const uint16_t* R, void* Y, void* ws, int32_t* err, cudaStream_t s) {
  switch (epi) {
    case FP_EPI_STORE: return launch_bt_t<MT, FP_EPI_STORE>(mw, mx, M, N, K, R, Y, ws, err, s);
    case FP_EPI_RESID: return launch_bt_t<MT, FP_EPI_RESID>(mw, mx, M, N, K, R, Y, ws, err, s);
    case FP_EPI_SWIGLU: return launch_bt_t<MT, FP_EPI_SWIGLU>(mw, mx, M, N, K, R, Y, ws, err, s);
    default: return launch_bt_t<MT, FP_EPI_F32>(mw, mx, M, N, K, R, Y, ws, err, s);
  }
}

cudaError_t launch_btc(int epi, const uint16_t* x, int M, int N, int K, const void* w, const uint16_t* residual,
                       void* y, void* ws, size_t ws_bytes, int32_t* err, cudaStream_t s) {
  if (!btc_ok(FP_W_BF16, epi, M, N, K)) return cudaErrorInvalidValue;
  if (!ws || ws_bytes < btc_ws_bytes(epi, M, N, K)) return cudaErrorInvalidValue;
  const int mt = M <= 32 ? 32 : 64;
  CUtensorMap mw, mx;
  // W [N][K] bf16, box [128 rows][64]; x [M][K] bf16, box [mt rows][64] (rows past M read zeros)
  if (!make_tensor_map(&mw, w, N, K, 2, kBtRows, kBtBK, 128)) return cudaErrorInvalidValue;
  if (!make_tensor_map(&mx, x, M, K, 2, mt, kBtBK, 128)) return cudaErrorInvalidValue;
  if (mt == 32) return launch_bt_m<32>(epi, mw, mx, M, N, K, residual, y, ws, err, s);
  return launch_bt_m<64>(epi, mw, mx, M, N, K, residual, y, ws, err, s);
}

}  // namespace fpk
