// Prefill linear with int8 / int4 weights, dequantised inside the tcgen05 GEMM.
//
// y[t][n] = sum_k x[t][k] deq(W)[n][k] for M > 64 tokens, the dense contraction
// of a decoder block's weight-only quantised linears (QKV, O, gate+up, down).
// The weights are the MMA's M side and the tokens its N side: a tile is 128
// weight rows x 256 tokens, so every 128 x 16 slab of dequantised weights
// feeds 256 tokens and the conversion costs half as many instructions per
// MMA cycle as it would with the weights on the 256-wide side.
//   warp 0      TMA producer of x: [256 tokens][64 k] bf16, 128-byte
//               swizzled, K-major, into stage s of a 4-stage ring
//               (xfull[s], bytes counted);
//   warp 1      allocates 512 TMEM columns (two 256-column fp32
//               accumulators) and, from one thread, issues tcgen05.mma
//               (M 128, N 256, K 16; A = weights, B = x, both from shared
//               memory); tcgen05.commit frees stage s (empty[s]) and hands a
//               full accumulator to the epilogue (tfull[b]);
//   warps 2-5   epilogue: tcgen05.ld of its 32 accumulator lanes (one weight
//               row, i.e. one output column, per thread), int8 row scale,
//               then store / residual add / fp32 store, or SwiGLU: the up
//               rows' warps pass their values to the gate rows' warps through
//               shared memory (uxfull / uxempty);
//   warps 6-13  dequantisers: each thread loads 16-byte pieces of code rows
//               from global memory four stages ahead (adjacent lanes read
//               adjacent pieces of one row), expands them to bf16 -- int8: the
//               code itself, exact, its row scale is applied in the epilogue;
//               int4: bf16((q - z) s), the product rounded once -- and stores
//               them as the A tile [128 rows][64 k] in the 128-byte-swizzled
//               K-major layout the MMA descriptor reads; fence.proxy.async and
//               one arrival per warp on afull[s].
// SwiGLU tiles hold 64 gate rows (lanes 0-63) and the matching 64 up rows
// (lanes 64-127), so one tile yields 64 output columns.
//
// Persistent: one CTA per SM takes tiles c, c + gridDim.x, ... in grouped
// order: GT token tiles (x rows that stay in L2) are swept over every weight
// row tile before the next group, so concurrently running CTAs share the
// same weight rows and x rows.
//
// Every mbarrier wait is bounded; past the limit the thread records error 2
// in the error word and the CTA stops, after its copies and MMAs in flight
// have completed and before TMEM is released.
#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace fpk {

constexpr int kWqRows = 128, kWqTok = 256, kWqBK = 64, kWqStages = 4;
constexpr int kWqEpiWarps = 4, kWqDeqWarps = 8;
constexpr int kWqAhead = 4;  // stages between a dequantiser's code load and its conversion
constexpr int kWqThreads = (2 + kWqEpiWarps + kWqDeqWarps) * 32;
constexpr uint32_t kWqABytes = kWqRows * kWqBK * 2;  // 16 KiB of bf16 weights
constexpr uint32_t kWqXBytes = kWqTok * kWqBK * 2;   // 32 KiB of bf16 x
constexpr uint32_t kWqStageBytes = kWqABytes + kWqXBytes;
constexpr uint32_t kWqXchgBytes = 32 * 64 * 4;  // SwiGLU: 32 tokens x 64 up rows, fp32
constexpr uint32_t kWqTmemCols = 512;
constexpr int kWqSmem = kWqStages * kWqStageBytes + 2 * kWqXchgBytes + 1024;

union WqBf2 {
  uint32_t u;
  __nv_bfloat162 h;
};

// One little-endian word of int4 codes (elements e0..e7 of a row, nibble i
// holding element (0,2,4,6,1,3,5,7)[i]) -> four bf16 pairs (q - z) s in
// element order.  (w >> 4i) & 0x000F000F | 0x43004300 is the bf16 pair
// (128 + q_2i, 128 + q_2i+1), exact; subtracting 128 + z is exact for integer
// codes; the multiplication by s rounds once, to nearest even.
FP_DEV void wq_int4_word(uint32_t w, uint32_t zz, uint32_t ss, uint32_t* out) {
  WqBf2 z2, s2;
  z2.u = zz;
  s2.u = ss;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    WqBf2 p;
    p.u = ((w >> (4 * i)) & 0x000F000Fu) | 0x43004300u;
    p.h = __hmul2(__hsub2(p.h, z2.h), s2.h);
    out[i] = p.u;
  }
}

// One word of four int8 codes -> two bf16 pairs q (exact).  Byte b of
// w ^ 0x80808080 is q_b + 128; placed under the exponent of 2^23 it gives the
// float 2^23 + q_b + 128, from which one subtraction leaves q_b exactly.  An
// integer of magnitude <= 127 is exact in bf16, so the upper half of its
// float is its bf16.
FP_DEV void wq_int8_word(uint32_t w, uint32_t* out) {
  const uint32_t u = w ^ 0x80808080u;
  float f[4];
#pragma unroll
  for (int b = 0; b < 4; ++b) f[b] = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7440 + b)) - 8388736.0f;
  out[0] = __byte_perm(__float_as_uint(f[0]), __float_as_uint(f[1]), 0x7632);
  out[1] = __byte_perm(__float_as_uint(f[2]), __float_as_uint(f[3]), 0x7632);
}

FP_DEV void st_shared16(uint32_t addr, const uint32_t* v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3])
               : "memory");
}

// Byte offset of 16-byte chunk c of row r in a K-major [rows][64] bf16 tile
// with the 128-byte swizzle: 8-row atoms of 1024 bytes, chunk c of row r at
// position c ^ (r % 8) within its 128-byte row.
FP_DEV uint32_t sw128_off(int r, int c) { return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4)); }

// Code pieces of one stage held by a dequantising thread: int4, one 16-byte
// piece (32 codes) and its group's scale and zero; int8, two pieces.
struct WqFrag {
  uint4 c[2];
  uint32_t s, z;
};

template <int WQ, int EPI>
__global__ void __launch_bounds__(kWqThreads, 1)
    gemm_wq_kernel(const __grid_constant__ CUtensorMap map_x, const uint8_t* __restrict__ codes, int M, int N, int K,
                   const uint16_t* __restrict__ scales, const uint16_t* __restrict__ zeros, const uint16_t* R,
                   void* Y, int GT, int32_t* err) {
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  constexpr int BRo = kWqRows / NR;                      // output columns per tile
  constexpr int UPT = WQ == FP_W_INT8 ? 2 : 1;           // 16-byte code pieces per thread and stage
  constexpr int PPR = WQ == FP_W_INT8 ? 4 : 2;           // pieces per row and stage
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t xfull[kWqStages], afull[kWqStages], empty[kWqStages], tfull[2], tempty[2];
  __shared__ uint64_t uxfull[2], uxempty[2], mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_word;
  volatile int* abort_flag = &abort_word;
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  float* xchg = (float*)(smem + kWqStages * kWqStageBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Nout = NR == 2 ? N / 2 : N;
  const int tiles_r = (Nout + BRo - 1) / BRo, tiles_t = (M + kWqTok - 1) / kWqTok;
  const int ntiles = tiles_r * tiles_t;
  const int kblocks = K / kWqBK + (K % kWqBK ? 1 : 0);
  auto tile_origin = [&](int t, int& r0, int& t0) {
    const int span = GT * tiles_r;
    const int first = (t / span) * GT;
    const int gs = min(GT, tiles_t - first);
    const int rem = t % span;
    t0 = (first + rem % gs) * kWqTok;
    r0 = (rem / gs) * BRo;
  };
  auto fail = [&]() {
    *abort_flag = 1;
    if (err) atomicExch(err, 2);
  };

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < kWqStages; ++s) {
      mbar_init(&xfull[s], 1);            // producer's expect_tx, completed by the bytes
      mbar_init(&afull[s], kWqDeqWarps);  // one arrival per dequantising warp
      mbar_init(&empty[s], 1);            // tcgen05.commit of the stage's MMAs
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kWqEpiWarps);
      mbar_init(&uxfull[b], 2);   // the two up-row warps wrote their values
      mbar_init(&uxempty[b], 2);  // the two gate-row warps read them
    }
    mbar_init(&mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                 "r"(kWqTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 0) {
    // ---------------- TMA producer of x
    if (lane == 0) {
      pdl_wait();  // x is the previous kernel's output
      int it = 0;
      for (int t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x) {
        int r0, t0;
        tile_origin(t, r0, t0);
        for (int kb = 0; kb < kblocks; ++kb, ++it) {
          const int s = it % kWqStages;
          if ((it >= kWqStages && !mbar_wait(&empty[s], ((it / kWqStages) & 1) ^ 1)) || *abort_flag) {
            fail();
            break;
          }
          mbar_expect_tx(&xfull[s], kWqXBytes);
          tma_load_2d(smem + s * kWqStageBytes + kWqABytes, &map_x, kb * kWqBK, t0, &xfull[s]);
        }
      }
      // copies still in flight land before the CTA leaves (their stages are its shared memory)
      for (int j = max(0, it - kWqStages); j < it; ++j) mbar_wait(&xfull[j % kWqStages], (j / kWqStages) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc(kWqRows, kWqTok);
      int it = 0, lt = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++lt) {
        const int acc = lt & 1;
        ok = mbar_wait(&tempty[acc], ((lt >> 1) & 1) ^ 1) && !*abort_flag;  // the epilogue drained it
        if (!ok) break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)acc * kWqTok;
        for (int kb = 0; kb < kblocks; ++kb, ++it) {
          const int s = it % kWqStages;
          const uint32_t par = (it / kWqStages) & 1;
          ok = mbar_wait(&xfull[s], par) && mbar_wait(&afull[s], par) && !*abort_flag;
          if (!ok) break;
          tc_fence_after();
          const uint32_t a = smem_u32(smem + s * kWqStageBytes);
          const uint32_t b = a + kWqABytes;
#pragma unroll
          for (int kk = 0; kk < kWqBK / 16; ++kk)
            tc_mma(d, sdesc(a + kk * 32), sdesc(b + kk * 32), idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          tc_commit(&empty[s]);  // stage s is free once these MMAs have read it
        }
        if (ok) tc_commit(&tfull[acc]);
      }
      if (!ok) fail();
      // every MMA issued has completed before TMEM is released
      tc_commit(&mma_done);
      mbar_wait(&mma_done, 0);
    }
  } else if (warp < 2 + kWqEpiWarps) {
    // ---------------- epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31
    const int q = warp & 3, lr = q * 32 + lane;
    pdl_wait();  // the residual and the output belong to the stream's order
    int lt = 0, ch = 0;  // local tile, SwiGLU exchange chunk (across tiles)
    for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++lt) {
      const int acc = lt & 1;
      int r0, t0;
      tile_origin(t, r0, t0);
      // the decision to stop is warp-uniform: tcgen05.ld below is warp-collective
      const bool got = __all_sync(0xffffffffu, mbar_wait(&tfull[acc], (lt >> 1) & 1));
      if (!got || __any_sync(0xffffffffu, *abort_flag != 0)) {
        if (lane == 0) fail();
        break;
      }
      tc_fence_after();
      // this lane's output column n and weight row wr
      const bool up = NR == 2 && lr >= 64;
      const int n = r0 + (up ? lr - 64 : lr);
      const bool valid = n < Nout;
      const int wr = up ? Nout + n : n;
      float sc = 1.f;
      if constexpr (WQ == FP_W_INT8) sc = valid ? bf2f(scales[wr]) : 0.f;
      const uint32_t tl = tmem + (uint32_t)acc * kWqTok + ((uint32_t)(q * 32) << 16);
      bool ok = true;
#pragma unroll 1
      for (int c0 = 0; c0 < kWqTok && t0 + c0 < M; c0 += 32, ++ch) {
        float v[32];
        tc_ld32(tl + c0, v);
        if constexpr (WQ == FP_W_INT8) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] *= sc;
        }
        const int cnt = min(32, M - (t0 + c0));
        if constexpr (NR == 2) {
          const int b = ch & 1;
          float* xb = xchg + b * (kWqXchgBytes / 4);
          if (up) {
            ok = __all_sync(0xffffffffu, ch < 2 || mbar_wait(&uxempty[b], ((ch >> 1) & 1) ^ 1));
            if (!ok) break;
#pragma unroll
            for (int i = 0; i < 32; ++i) xb[i * 64 + (lr - 64)] = v[i];
            __syncwarp();
            if (lane == 0) mbar_arrive(&uxfull[b]);
          } else {
            ok = __all_sync(0xffffffffu, mbar_wait(&uxfull[b], (ch >> 1) & 1));
            if (!ok) break;
            float u[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) u[i] = xb[i * 64 + lr];
            __syncwarp();
            if (lane == 0) mbar_arrive(&uxempty[b]);
            if (valid) {
              uint16_t* y = (uint16_t*)Y + (long long)(t0 + c0) * Nout + n;
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (i < cnt) y[(long long)i * Nout] = f2bf(silu(v[i]) * u[i]);
            }
          }
        } else if (valid) {
          const long long o = (long long)(t0 + c0) * Nout + n;
          if constexpr (EPI == FP_EPI_F32) {
            float* y = (float*)Y + o;
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (i < cnt) y[(long long)i * Nout] = v[i];
          } else if constexpr (EPI == FP_EPI_RESID) {
            uint16_t* y = (uint16_t*)Y + o;
#pragma unroll
            for (int h = 0; h < 32; h += 16) {  // 16 residual loads in flight at a time
              float r[16];
#pragma unroll
              for (int i = 0; i < 16; ++i) r[i] = h + i < cnt ? bf2f(R[o + (long long)(h + i) * Nout]) : 0.f;
#pragma unroll
              for (int i = 0; i < 16; ++i)
                if (h + i < cnt) y[(long long)(h + i) * Nout] = f2bf(r[i] + v[h + i]);
            }
          } else {
            uint16_t* y = (uint16_t*)Y + o;
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (i < cnt) y[(long long)i * Nout] = f2bf(v[i]);
          }
        }
      }
      if (!ok) {
        if (lane == 0) fail();
        break;
      }
      // this warp's reads of the accumulator are done: hand it back to the MMA thread
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
  } else {
    // ---------------- dequantisers: thread dt owns pieces dt + 256 j of every stage
    // (a fixed A row and 16-byte piece of the row's codes), so the shared-memory
    // offsets are computed once and a stage costs one pointer step per piece
    constexpr int CPU = WQ == FP_W_INT8 ? 2 : 4;  // 16-byte bf16 chunks per piece
    constexpr long long STEP = WQ == FP_W_INT8 ? kWqBK : kWqBK / 2;  // code bytes per row and stage
    const int dt = threadIdx.x - (2 + kWqEpiWarps) * 32;
    const int G = K / 128;  // int4 groups per row
    const long long row_bytes = WQ == FP_W_INT8 ? (long long)K : (long long)K / 2;
    const int total = ((ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x) * kblocks;
    int ar[UPT], pc[UPT];
    uint32_t soff[UPT][CPU];
#pragma unroll
    for (int j = 0; j < UPT; ++j) {
      const int u = dt + 256 * j;
      ar[j] = u / PPR;
      pc[j] = u % PPR;
#pragma unroll
      for (int h = 0; h < CPU; ++h) soff[j][h] = sw128_off(ar[j], CPU * pc[j] + h);
    }
    // load cursor: the next stage to fetch, its tile's code rows (null: a row
    // past the matrix, which converts to zeros)
    int l_it = 0, l_lt = -1, l_kb = kblocks;
    const uint8_t* cp[UPT];
    const uint16_t* sp = nullptr;
    const uint16_t* zp = nullptr;
    auto load = [&](WqFrag& f) {
      if (l_it >= total) return;
      if (l_kb == kblocks) {  // next tile: its code rows
        l_kb = 0;
        ++l_lt;
        int r0, t0;
        tile_origin((int)blockIdx.x + l_lt * (int)gridDim.x, r0, t0);
#pragma unroll
        for (int j = 0; j < UPT; ++j) {
          int wr;
          if (NR == 2) {
            const int n = r0 + (ar[j] & 63);
            wr = n < Nout ? (ar[j] < 64 ? n : Nout + n) : -1;
          } else {
            wr = r0 + ar[j] < Nout ? r0 + ar[j] : -1;
          }
          cp[j] = wr >= 0 ? codes + (long long)wr * row_bytes + pc[j] * 16 : nullptr;
          if (WQ == FP_W_INT4_G128 && j == 0) {
            sp = wr >= 0 ? scales + (long long)wr * G : nullptr;
            zp = wr >= 0 ? zeros + (long long)wr * G : nullptr;
          }
        }
      }
#pragma unroll
      for (int j = 0; j < UPT; ++j) {
        const bool in = cp[j] != nullptr && (WQ != FP_W_INT8 || l_kb * kWqBK + pc[j] * 16 < K);
        f.c[j] = in ? ld_nc16(cp[j] + l_kb * STEP) : make_uint4(0u, 0u, 0u, 0u);
      }
      if (WQ == FP_W_INT4_G128) {
        f.s = sp ? __ldg(sp + (l_kb >> 1)) : 0u;
        f.z = zp ? __ldg(zp + (l_kb >> 1)) : 0u;
      }
      ++l_kb;
      ++l_it;
    };
    const uint32_t smem0 = smem_u32(smem);
    auto process = [&](int it, const WqFrag& f) -> bool {
      if (it >= total) return true;
      const int s = it % kWqStages;
      const bool free_ = it < kWqStages || mbar_wait(&empty[s], ((it / kWqStages) & 1) ^ 1);
      if (!__all_sync(0xffffffffu, free_) || __any_sync(0xffffffffu, *abort_flag != 0)) return false;
      const uint32_t a = smem0 + s * kWqStageBytes;
      if constexpr (WQ == FP_W_INT8) {
#pragma unroll
        for (int j = 0; j < UPT; ++j) {
          // 16 codes: chunk 2 pc holds codes 0-7, chunk 2 pc + 1 codes 8-15
          uint32_t o[4];
          wq_int8_word(f.c[j].x, o);
          wq_int8_word(f.c[j].y, o + 2);
          st_shared16(a + soff[j][0], o);
          wq_int8_word(f.c[j].z, o);
          wq_int8_word(f.c[j].w, o + 2);
          st_shared16(a + soff[j][1], o);
        }
      } else {
        // 32 codes: chunks 4 pc .. 4 pc + 3, one code word each
        const uint32_t zb = f2bf(128.f + bf2f((uint16_t)f.z));
        const uint32_t zz = zb | (zb << 16), ss = f.s | (f.s << 16);
        uint32_t o[4];
        wq_int4_word(f.c[0].x, zz, ss, o);
        st_shared16(a + soff[0][0], o);
        wq_int4_word(f.c[0].y, zz, ss, o);
        st_shared16(a + soff[0][1], o);
        wq_int4_word(f.c[0].z, zz, ss, o);
        st_shared16(a + soff[0][2], o);
        wq_int4_word(f.c[0].w, zz, ss, o);
        st_shared16(a + soff[0][3], o);
      }
      fence_proxy_async();  // the generic-proxy stores reach the MMA's async proxy
      __syncwarp();
      if (lane == 0) mbar_arrive(&afull[s]);
      return true;
    };
    // codes are loaded kWqAhead stages ahead of their conversion: a register
    // ring, indexed by constants once the inner loop is unrolled
    WqFrag f[kWqAhead + 1];
#pragma unroll
    for (int i = 0; i < kWqAhead; ++i) load(f[i]);
    bool ok = true;
    for (int it = 0; it < total && ok; it += kWqAhead + 1) {
#pragma unroll
      for (int i = 0; i <= kWqAhead; ++i) {
        load(f[(i + kWqAhead) % (kWqAhead + 1)]);
        ok = process(it + i, f[i]);
        if (!ok) break;
      }
    }
    if (!ok && lane == 0) fail();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kWqTmemCols) : "memory");
  }
}

// ------------------------------------------------------------------ host side
bool gemm_wq_ok(int wquant, int epi, int M, int N, int K, const void* x, const void* codes) {
  if (M <= 64 || N < 1 || K < 16 || K % 8 != 0 || !tensor_maps_available()) return false;
  if (epi == FP_EPI_SWIGLU && N % 2 != 0) return false;
  if (((uintptr_t)x & 15) || ((uintptr_t)codes & 15)) return false;
  if (wquant == FP_W_INT8) return K % 16 == 0;
  if (wquant == FP_W_INT4_G128) return K % 128 == 0;
  return false;
}

template <int WQ, int EPI>
static cudaError_t launch_wq_t(const CUtensorMap& mx, const uint8_t* codes, int M, int N, int K,
                               const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* Y,
                               int32_t* err, cudaStream_t s) {
  auto kern = gemm_wq_kernel<WQ, EPI>;
  static std::atomic<unsigned long long> attr{0};
  FP_CUDA_TRY(smem_limit_once(kern, kWqSmem, &attr));
  constexpr int BRo = EPI == FP_EPI_SWIGLU ? kWqRows / 2 : kWqRows;
  const int Nout = EPI == FP_EPI_SWIGLU ? N / 2 : N;
  const long long tiles = (long long)((Nout + BRo - 1) / BRo) * ((M + kWqTok - 1) / kWqTok);
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        sms <= 0)
      sms = 152;
  }
  // token tiles per sweep: their x rows (256 x K bf16 each) within about 64 MB of L2
  const int GT = (int)std::max<long long>(1, std::min<long long>(16, (64ll << 20) / ((long long)kWqTok * K * 2)));
  const dim3 grid((unsigned)std::min<long long>(tiles, sms));
  return launch(kern, grid, dim3(kWqThreads), (size_t)kWqSmem, s, mx, codes, M, N, K, scales, zeros, R, Y, GT, err);
}

template <int WQ>
static cudaError_t launch_wq_w(int epi, const CUtensorMap& mx, const uint8_t* codes, int M, int N, int K,
                               const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* Y,
                               int32_t* err, cudaStream_t s) {
  switch (epi) {
    case FP_EPI_STORE: return launch_wq_t<WQ, FP_EPI_STORE>(mx, codes, M, N, K, scales, zeros, R, Y, err, s);
    case FP_EPI_RESID: return launch_wq_t<WQ, FP_EPI_RESID>(mx, codes, M, N, K, scales, zeros, R, Y, err, s);
    case FP_EPI_SWIGLU: return launch_wq_t<WQ, FP_EPI_SWIGLU>(mx, codes, M, N, K, scales, zeros, R, Y, err, s);
    default: return launch_wq_t<WQ, FP_EPI_F32>(mx, codes, M, N, K, scales, zeros, R, Y, err, s);
  }
}

cudaError_t launch_gemm_wq(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                           const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y,
                           int32_t* err, cudaStream_t s) {
  if (!gemm_wq_ok(wquant, epi, M, N, K, x, codes)) return cudaErrorInvalidValue;
  CUtensorMap mx;
  // x [M][K] bf16, box [256 tokens][64]
  if (!make_tensor_map(&mx, x, M, K, 2, kWqTok, kWqBK, 128)) return cudaErrorInvalidValue;
  const uint8_t* c = (const uint8_t*)codes;
  if (wquant == FP_W_INT8) return launch_wq_w<FP_W_INT8>(epi, mx, c, M, N, K, scales, zeros, residual, y, err, s);
  return launch_wq_w<FP_W_INT4_G128>(epi, mx, c, M, N, K, scales, zeros, residual, y, err, s);
}

}  // namespace fpk
