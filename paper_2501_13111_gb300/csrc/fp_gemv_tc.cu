// Decode linear for int4 group-128 (and int8 per-channel) weights at 17-64
// tokens on the tcgen05 tensor cores.
//
// y[m][n] = sum_k x[m][k] (q[n][k] - z[n][g]) s[n][g], g = k / 128, the
// weight-only linear of a decoder block (QKV, O, gate+up, down) while the
// decode batch is large enough that int4 dequantisation plus the legacy
// mma.sync rate, not HBM, bound the CUDA-core GEMV (two weights per byte,
// 2 M flop per weight).  The weights are the A operand (128 rows, one TMEM
// lane each) and the tokens the N dimension of tcgen05.mma (M 128, N =
// tokens rounded up to 32 or 64, K 16):
//   warps 0-15  dequantise, in two teams of eight that take alternate
//               items (KI consecutive k of a row tile; SwiGLU: of the gate
//               and of the up tile): warp w owns TMEM lanes 32 (w % 4) .. +31
//               (one weight row per thread) and the first or second half of
//               the item's k (SwiGLU: the gate or the up row).  Each thread
//               streams its own codes through a private cp.async ring in
//               shared memory (no cross-warp handshake),
//               forms bf16((q - z) s) -- exactly the prefill expansion --
//               and stores them into an A slot of TMEM (tcgen05.st, two K
//               elements per 32-bit column); afull / aempty hand the slots
//               to the MMA thread and back;
//   warp 16     TMA producer of x ([N][KI] bf16 per item as [N][64]
//               128-byte-swizzled boxes, rows past M zero-filled) into a ring
//               whose stage a goes with A slot a: afull[a] completes when the
//               team's warps have stored the slot and the x bytes have
//               landed, and one commit of the MMAs frees both (aempty[a]), so
//               the MMA thread waits once and commits once per item;
//   warps 17-18 issue the MMAs (A from TMEM, B = x from shared memory) into
//               fp32 TMEM accumulators, each its own chains (SwiGLU: one
//               matrix each); warp 17 also allocates the 512 TMEM columns.
// MMAs (M 128, N <= 64, K 16) into one accumulator follow each other at
// about 50 cycles, far above their math (N / 2 cycles), while MMAs into
// different accumulators overlap: the k-steps of each matrix are spread
// round-robin over 2-4 accumulators ("chains"), summed in the epilogue.
// The (row tile, item) pairs are split into equal contiguous ranges, one
// per SM (stream-K, as the CUDA-core GEMV): a CTA whose range covers a whole
// row tile runs the epilogue itself; otherwise each of its sixteen warps
// writes fp32 partials of its 32 rows x a quarter of the tokens, and the
// last CTA to finish that slice (a ticket per slice) sums them in CTA order
// and runs the epilogue -- residual add, SwiGLU, bf16 or fp32 store.
//
// int8 per-channel weights, y[m][n] = s[n] sum_k x[m][k] q[n][k], take the
// same pipeline with items of 128 k (64 k of each matrix with SwiGLU): the
// codes are widened exactly to bf16 (the integer q) and the row scale
// multiplies the fp32 sums in the epilogue.
//
// Every mbarrier wait is bounded; past the limit the thread records error 2
// in the error word, the CTA stops and releases TMEM after its copies and
// MMAs have completed.
#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace fpk {

// per-thread cp.async ring depth, one (own) item per stage; with 16 KB items
// 3 stages measured 1-4 % faster than 4 (70B shapes at 32 tokens) and 5 slower
constexpr int kQ4CodeStages = 3;
constexpr int kQ4DeqWarps = 16;
constexpr int kQ4MmaWarps = 2;  // MMA issuers, each with its own accumulators
constexpr int kQ4Threads = (kQ4DeqWarps + 1 + kQ4MmaWarps) * 32;
constexpr uint32_t kQ4TmemCols = 512;
constexpr int kQ4Rows = 128;
constexpr int kQ4MinSmem = 116 * 1024;  // above half an SM: one CTA (and one TMEM owner) per SM

// An item is KI consecutive k of one row tile (of the gate and the up tile
// with SwiGLU), 8 or 16 KB of codes: int4 one 128-k group, or two where K is
// a multiple of 256 and there is no SwiGLU; int8 128 k, or 64 k of each
// matrix with SwiGLU.  Larger items halve the hand-offs per byte.
template <int MT, int NR, int WQ, int KI>
struct Q4Geom {
  static_assert(WQ == FP_W_INT8 || KI % 128 == 0, "int4 items hold whole groups");
  static constexpr int kRowBytes = WQ == FP_W_INT8 ? KI : KI / 2;  // codes of one row of an item
  // each thread takes every other item: its row's codes of the item (SwiGLU:
  // of the gate or the up row), otherwise half of them
  static constexpr int kThreadBytes = NR == 2 ? kRowBytes : kRowBytes / 2;
  static constexpr int kChunks = kThreadBytes / 16;     // 16-byte code chunks per thread and item
  static_assert(kChunks == 2 || kChunks == 4, "two or four chunks per thread");
  static_assert(WQ == FP_W_INT4_G128 || kChunks == 4, "int8: one 32-column TMEM store per thread and item");
  static constexpr int kCodeBytes = kQ4DeqWarps * 32 * kChunks * 16;  // one ring stage, all threads
  static constexpr int kXBytes = MT * KI * 2;            // x [MT][KI] bf16 as [MT][64] boxes
  // independent accumulation chains per matrix
  static constexpr int kChains = MT == 64 ? 2 / NR : 4 / NR;
  static constexpr int kDCols = NR * kChains * MT;       // fp32 accumulators
  static constexpr int kACols = NR * KI / 2;             // the item's bf16 pairs
  static constexpr int kASlots = std::min(6, ((int)kQ4TmemCols - kDCols) / kACols);
  // x stage a travels with A slot a: one barrier per item says both are ready
  // and one commit frees both
  static constexpr int kXStages = kASlots;
  static constexpr int kSmem = kQ4CodeStages * kCodeBytes + kXStages * kXBytes + 1024;
  static_assert(kASlots >= 2 && kDCols + kASlots * kACols <= (int)kQ4TmemCols, "TMEM budget");
  static_assert(kCodeBytes % 1024 == 0 && kXBytes % 1024 == 0, "x stages stay 1024-byte aligned");
  static_assert(kSmem <= 227 * 1024, "shared memory");
};

// 16-byte asynchronous global -> shared copy (L2 only) and its group fences.
FP_DEV void q4_cp16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem)), "l"(gmem) : "memory");
}
FP_DEV void q4_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
FP_DEV void q4_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// V consecutive bf16 (V = 8, 4, 2 or 1, aligned to V elements) in a uint4.
FP_DEV uint4 ld_groups(const uint16_t* p, int V) {
  if (V == 8) return __ldg(reinterpret_cast<const uint4*>(p));
  if (V == 4) {
    const uint2 t = __ldg(reinterpret_cast<const uint2*>(p));
    return make_uint4(t.x, t.y, 0u, 0u);
  }
  if (V == 2) return make_uint4(__ldg(reinterpret_cast<const unsigned int*>(p)), 0u, 0u, 0u);
  return make_uint4((uint32_t)__ldg(reinterpret_cast<const unsigned short*>(p)), 0u, 0u, 0u);
}

FP_DEV uint32_t bf16_at(const uint4& v, int j) {
  const int w = j >> 1;
  const uint32_t x = w == 0 ? v.x : w == 1 ? v.y : w == 2 ? v.z : v.w;
  return (j & 1) ? (x >> 16) : (x & 0xFFFFu);
}

union Bf2 {
  uint32_t u;
  __nv_bfloat162 h;
};

// One packed word of int4 codes (elements 8j .. 8j+7; nibbles i and i + 4
// hold elements 2i and 2i + 1) -> four bf16 pairs (q - z) s in element order.
// bf16(128 + q) is formed exactly by the exponent trick; subtracting
// bf16(128 + z) is exact for integer z in [0, 15]; the product is rounded
// once, to nearest even.
FP_DEV void deq_word(uint32_t w, uint32_t zz, uint32_t ss, uint32_t* out) {
  Bf2 z2, s2;
  z2.u = zz;
  s2.u = ss;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    Bf2 p;
    p.u = ((w >> (4 * i)) & 0x000F000Fu) | 0x43004300u;
    p.h = __hmul2(__hsub2(p.h, z2.h), s2.h);
    out[i] = p.u;
  }
}

// One word of four int8 codes -> two bf16 pairs q (exact).  Byte b of
// w ^ 0x80808080 is q_b + 128; placed under the exponent of 2^23 it gives the
// float 2^23 + q_b + 128, from which one subtraction leaves q_b exactly, and
// an integer of magnitude <= 127 is exact in bf16: the float's upper half.
FP_DEV void i8_word(uint32_t w, uint32_t* out) {
  const uint32_t u = w ^ 0x80808080u;
  float f[4];
#pragma unroll
  for (int b = 0; b < 4; ++b) f[b] = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7440 + b)) - 8388736.0f;
  out[0] = __byte_perm(__float_as_uint(f[0]), __float_as_uint(f[1]), 0x7632);
  out[1] = __byte_perm(__float_as_uint(f[2]), __float_as_uint(f[3]), 0x7632);
}

FP_DEV long long q4_cta_of(long long i, long long C, long long total) { return ((i + 1) * C - 1) / total; }

template <int MT, int EPI, int WQ, int KI>
__global__ void __launch_bounds__(kQ4Threads, 1)
    gemv_q4tc_kernel(const __grid_constant__ CUtensorMap map_x, const uint8_t* __restrict__ codes, int M, int N,
                     const uint16_t* __restrict__ scales, const uint16_t* __restrict__ zeros, const uint16_t* R,
                     void* Y, long long total, int S, int V, float* __restrict__ ws, unsigned* __restrict__ counters,
                     int32_t* err) {
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  using G = Q4Geom<MT, NR, WQ, KI>;
  constexpr bool I4 = WQ == FP_W_INT4_G128;
  constexpr int GPI = I4 ? KI / 128 : 1;  // int4: groups per item
  constexpr int CS = kQ4CodeStages, XS = G::kXStages, NA = G::kASlots, MQ = MT / 4, DW = kQ4DeqWarps;
  constexpr int NCH = G::kChains, CK = G::kChunks;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  static_assert(XS == NA, "x stages and A slots share their barriers");
  __shared__ uint64_t afull[NA], aempty[NA], dfull, dempty, mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_word;
  volatile int* abort_flag = &abort_word;
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* x_ring = smem;                               // 1024-byte aligned for the 128-byte swizzle
  uint8_t* code_ring = smem + XS * G::kXBytes;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Nout = NR == 2 ? N / 2 : N;
  const long long C = gridDim.x, c = blockIdx.x;
  const long long begin = c * total / C, end = (c + 1) * total / C;
  const int L = (int)(end - begin);
  const int SI = S * 128 / KI;  // items per row tile (S: 128-k groups per row)
  auto fail = [&]() {
    *abort_flag = 1;
    if (err) atomicExch(err, 2);
  };

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int a = 0; a < NA; ++a) {
      // the eight warps of the item's team stored its A columns, and the x
      // producer's expect_tx, completed by the bytes of the item's x
      mbar_init(&afull[a], DW / 2 + 1);
      mbar_init(&aempty[a], kQ4MmaWarps);  // tcgen05.commit of the MMAs that read slot and stage
    }
    mbar_init(&dfull, kQ4MmaWarps);
    mbar_init(&dempty, DW);
    mbar_init(&mma_done, kQ4MmaWarps);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == DW + 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                 "r"(kQ4TmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == DW) {
    // ---------------- TMA producer of x
    if (lane == 0) {
      pdl_wait();  // x is the previous kernel's output
      int issued = 0;
      int g = (int)(begin % SI);
      for (int q = 0; q < L; ++q, g = g + 1 == SI ? 0 : g + 1) {
        const int s = q % XS;
        if (q >= XS && (!mbar_wait_sleep(&aempty[s], ((q / XS) & 1) ^ 1) || *abort_flag)) {
          fail();
          break;
        }
        uint8_t* xs = x_ring + s * G::kXBytes;
        mbar_expect_tx(&afull[s], G::kXBytes);
#pragma unroll
        for (int bx = 0; bx < KI / 64; ++bx) tma_load_2d(xs + bx * MT * 128, &map_x, g * KI + bx * 64, 0, &afull[s]);
        issued = q + 1;
      }
      // copies still in flight land before the CTA leaves (their stages are its
      // shared memory); after an abort the phase may never complete, and the
      // bounded wait then outlasts the copies
      for (int j = max(0, issued - XS); j < issued; ++j) mbar_wait(&afull[j % XS], (j / XS) & 1);
    }
  } else if (warp > DW) {
    // ---------------- MMA issuers: SwiGLU, one per matrix; otherwise even / odd k-steps
    const int mw = warp - DW - 1;
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc(kQ4Rows, MT);
      int seg = 0;
      bool ok = true;
      int g = (int)(begin % SI);
      for (int q = 0; q < L; ++q, g = g + 1 == SI ? 0 : g + 1) {
        const bool first = q == 0 || g == 0, last = g == SI - 1 || q == L - 1;
        const int s = q % XS, a = q % NA;
        if (first && seg > 0) ok = mbar_wait(&dempty, (seg - 1) & 1);  // the epilogue has read D
        ok = ok && mbar_wait(&afull[a], (q / NA) & 1) && !*abort_flag;  // A slot and x stage
        if (!ok) break;
        tc_fence_after();
        const uint64_t xd = sdesc(smem_u32(x_ring + s * G::kXBytes));
        const uint32_t ta = tmem + G::kDCols + a * G::kACols;
        // k-step kk of matrix r goes to chain kk % NCH of that matrix: consecutive
        // MMAs of one issuer never share an accumulator, and the two issuers'
        // chains are disjoint
#pragma unroll
        for (int kk = 0; kk < KI / 16; ++kk) {
          const int r = NR == 2 ? mw : 0;
          if (NR == 1 && (kk & 1) != mw) continue;
          // descriptor start addresses count 16-byte units; k-step kk reads A
          // columns 8 kk .. +7 (of matrix r) and x box kk / 4
          tc_mma_ts(tmem + (r * NCH + kk % NCH) * MT, ta + r * (KI / 2) + kk * 8,
                    xd + (uint64_t)(((kk >> 2) * MT * 128 + (kk & 3) * 32) >> 4), idesc, (first && kk < NCH) ? 0u : 1u);
        }
        tc_commit(&aempty[a]);  // A slot a and x stage a have been read
        if (last) {
          tc_commit(&dfull);
          ++seg;
        }
      }
      if (!ok) fail();
      // every MMA issued has completed before TMEM is released
      tc_commit(&mma_done);
      mbar_wait(&mma_done, 0);
    }
  } else {
    // ---------------- dequantise (+ epilogue)
    // two teams of eight warps take alternate items, so one team computes
    // while the other waits; within a team warp w owns TMEM lanes
    // 32 (w % 4) .. +31 and, SwiGLU, the gate or the up rows, otherwise the
    // first or second half of the item's k (int4 with two groups per item:
    // the first or the second group)
    const int qd = warp & 3, team = warp >> 3, half = (warp >> 2) & 1, lr = qd * 32 + lane;
    const int pt = warp >> 2;  // epilogue: tokens [pt MQ, (pt + 1) MQ)
    const int rm = NR == 2 ? half : 0;
    const int gsel = (I4 && GPI == 2) ? half : 0;                   // int4: this warp's group of the item
    const int tboff = NR == 1 ? half * G::kThreadBytes : 0;         // this warp's bytes of the item's row
    const int acol = NR == 2 ? rm * (KI / 2) : half * (KI / 4);
    const uint32_t lane_base = tmem + ((uint32_t)(qd * 32) << 16);
    const long long row_bytes = (long long)SI * G::kRowBytes;

    // ---- this thread's code ring: its n-th own item (team + 2 n) in stage
    // n % CS, chunk i at [stage][i][thread] (a warp's loads of one chunk are
    // 512 contiguous bytes)
    uint8_t* my_ring = code_ring + (size_t)threadIdx.x * 16;
    const int own = (L - team + 1) / 2;  // items this team takes
    int ib = (int)((begin + team) / SI), ig = (int)((begin + team) % SI);  // (row tile, item) of the next copy
    const uint8_t* src = nullptr;
    auto set_src = [&]() {
      const long long rr = min(ib * kQ4Rows + lr, Nout - 1) + rm * Nout;
      src = codes + rr * row_bytes + tboff;
    };
    if (own > 0) set_src();
    auto issue = [&](int n) {  // called for n = 0, 1, 2, ... in order
      if (n < own) {
        uint8_t* d = my_ring + (size_t)(n % CS) * G::kCodeBytes;
#pragma unroll
        for (int i = 0; i < CK; ++i) q4_cp16(d + i * (DW * 32 * 16), src + (long long)ig * G::kRowBytes + i * 16);
        ig += 2;
        if (ig >= SI) {
          while (ig >= SI) ig -= SI, ++ib;
          if (n + 1 < own) set_src();
        }
      }
      q4_commit();
    };
    // the weights are constant: the first stages go out before the previous kernel ends
#pragma unroll 1
    for (int n = 0; n < CS - 1; ++n) issue(n);

    // int4: scales and zeros of the row, V groups (VI items) per load, one
    // chunk ahead (S % V == 0, so a chunk never crosses a row tile); int8 has
    // one scale per row, applied in the epilogue
    const int VI = I4 ? V / GPI : 1;
    uint4 s_cur = make_uint4(0u, 0u, 0u, 0u), z_cur = s_cur, s_nxt = s_cur, z_nxt = s_cur;
    auto load_chunk = [&](int bb, int g0, uint4& sv, uint4& zv) {  // g0: first item of the chunk
      if constexpr (I4) {
        const long long idx = (long long)(min(bb * kQ4Rows + lr, Nout - 1) + rm * Nout) * S + (long long)g0 * GPI;
        sv = ld_groups(scales + idx, V);
        zv = ld_groups(zeros + idx, V);
      }
    };
    // (row tile, item) of the current item and its place j in the chunk of VI
    // items, advanced without divisions
    int b = (int)(begin / SI), g = (int)(begin % SI), j = g % VI;
    load_chunk(b, g - j, s_cur, z_cur);
    auto prefetch_next = [&](long long p_next, int bb, int g0) {  // the chunk starting at item p_next
      if (g0 == SI) g0 = 0, ++bb;
      if (p_next < end) load_chunk(bb, g0, s_nxt, z_nxt);
    };
    prefetch_next(begin - j + VI, b, g - j + VI);
    pdl_wait();
    int seg = 0;
    for (int q = 0; q < L; ++q) {
      const long long p = begin + q;
      if (q > 0) {
        if (++g == SI) g = 0, ++b;
        if (++j == VI) {
          j = 0;
          s_cur = s_nxt;
          z_cur = z_nxt;
          prefetch_next(p + VI, b, g + VI);
        }
      }
      const bool last = g == SI - 1 || q == L - 1;
      if ((q & 1) == team) {
        const int n = q >> 1, a = q % NA;
        q4_wait<CS - 2>();  // this thread's copies of its n-th item have landed
        uint4 wv[CK];
#pragma unroll
        for (int i = 0; i < CK; ++i)
          wv[i] = *reinterpret_cast<const uint4*>(my_ring + (size_t)(n % CS) * G::kCodeBytes + i * (DW * 32 * 16));
        issue(n + CS - 1);  // refills the stage read one own item ago

        const uint32_t ta = lane_base + G::kDCols + a * G::kACols + acol;
        bool ok = true;
        auto slot_free = [&]() {  // the first columns are converted while the slot drains
          ok = mbar_wait_sleep(&aempty[a], ((q / NA) & 1) ^ 1);
          ok = __all_sync(0xffffffffu, ok) && !__any_sync(0xffffffffu, *abort_flag != 0);
          if (ok) tc_fence_after();
          return ok;
        };
        if constexpr (I4) {
          const uint32_t sb = bf16_at(s_cur, j * GPI + gsel);
          const uint32_t zb = f2bf(128.f + bf2f((uint16_t)bf16_at(z_cur, j * GPI + gsel)));
          const uint32_t ss = sb | (sb << 16), zz = zb | (zb << 16);
#pragma unroll
          for (int h2 = 0; h2 < CK / 2; ++h2) {  // 32 columns (two chunks) per store
            uint32_t av[32];
#pragma unroll
            for (int i = 0; i < 2; ++i) {
              const uint4 w = wv[2 * h2 + i];
              deq_word(w.x, zz, ss, av + i * 16);
              deq_word(w.y, zz, ss, av + i * 16 + 4);
              deq_word(w.z, zz, ss, av + i * 16 + 8);
              deq_word(w.w, zz, ss, av + i * 16 + 12);
            }
            if (h2 == 0 && !slot_free()) break;
            tc_st32(ta + h2 * 32, av);
          }
        } else {
          uint32_t av[32];  // four chunks of 16 codes: 32 columns of bf16 pairs
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            i8_word(wv[i].x, av + i * 8);
            i8_word(wv[i].y, av + i * 8 + 2);
            i8_word(wv[i].z, av + i * 8 + 4);
            i8_word(wv[i].w, av + i * 8 + 6);
          }
          if (slot_free()) tc_st32(ta, av);
        }
        if (!ok) {
          if (lane == 0) fail();
          break;
        }
        tc_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&afull[a]);
      }
      if (!last) continue;

      // ---- the CTA's part of row tile b is accumulated: this warp takes tokens [m0, m0 + MQ)
      bool ok = mbar_wait_sleep(&dfull, seg & 1);
      if (!__all_sync(0xffffffffu, ok) || __any_sync(0xffffffffu, *abort_flag != 0)) {
        if (lane == 0) fail();
        break;
      }
      tc_fence_after();
      const int m0 = pt * MQ;
      uint32_t dv[NR][MQ];
#pragma unroll
      for (int r = 0; r < NR; ++r) {
        tc_ld<MQ>(lane_base + r * NCH * MT + m0, dv[r]);
#pragma unroll
        for (int ch = 1; ch < NCH; ++ch) {  // the chains' sum, in chain order
          uint32_t e[MQ];
          tc_ld<MQ>(lane_base + (r * NCH + ch) * MT + m0, e);
#pragma unroll
          for (int i = 0; i < MQ; ++i) dv[r][i] = __float_as_uint(__uint_as_float(dv[r][i]) + __uint_as_float(e[i]));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&dempty);
      ++seg;

      const int row = b * kQ4Rows + lr;
      // int8: the row scales (gate and up rows with SwiGLU) multiply the sums
      float sg = 1.f, su = 1.f;
      if constexpr (!I4) {
        const int rc = min(row, Nout - 1);
        sg = bf2f(scales[rc]);
        su = bf2f(scales[(NR - 1) * Nout + rc]);
      }
      // r: the residual R[m][row], read before any store (R may be Y itself)
      auto resid = [&](int m) {
        return (EPI == FP_EPI_RESID && m < M && row < Nout) ? bf2f(R[(long long)m * Nout + row]) : 0.f;
      };
      auto finish = [&](int m, float v, float u, float r) {
        const long long o = (long long)m * Nout + row;
        v *= sg;
        u *= su;
        if constexpr (EPI == FP_EPI_STORE) ((uint16_t*)Y)[o] = f2bf(v);
        else if constexpr (EPI == FP_EPI_RESID) ((uint16_t*)Y)[o] = f2bf(r + v);
        else if constexpr (EPI == FP_EPI_SWIGLU) ((uint16_t*)Y)[o] = f2bf(silu(v) * u);
        else ((float*)Y)[o] = v;
      };
      const long long c0 = q4_cta_of((long long)b * SI, C, total);
      const long long c1 = q4_cta_of((long long)(b + 1) * SI - 1, C, total);
      if (c0 == c1) {
#pragma unroll
        for (int i0 = 0; i0 < MQ; i0 += 8) {
          float rv[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) rv[i] = resid(m0 + i0 + i);
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (m0 + i0 + i < M && row < Nout)
              finish(m0 + i0 + i, __uint_as_float(dv[0][i0 + i]), __uint_as_float(dv[NR - 1][i0 + i]), rv[i]);
        }
        continue;
      }
      // partial slot b + c: distinct for every (row tile, CTA) pair that meets
      const size_t slot = (size_t)M * NR * kQ4Rows;
      float* part = ws + (size_t)(b + c) * slot;
#pragma unroll
      for (int i = 0; i < MQ; ++i)
        if (m0 + i < M)
#pragma unroll
          for (int r = 0; r < NR; ++r) part[((size_t)(m0 + i) * NR + r) * kQ4Rows + lr] = __uint_as_float(dv[r][i]);
      __threadfence();
      __syncwarp();
      unsigned t = 0;
      if (lane == 0) t = atomicAdd(&counters[b * DW + warp], 1u);
      t = __shfl_sync(0xffffffffu, t, 0);
      if (t != (unsigned)(c1 - c0)) continue;
      __threadfence();
      // the sum over the CTAs in CTA order (deterministic), eight tokens' loads
      // in flight per CTA rather than one
      const int cnt = (int)(c1 - c0) + 1;
      const float* p0 = ws + (size_t)(b + c0) * slot + (size_t)m0 * NR * kQ4Rows + lr;
#pragma unroll
      for (int i0 = 0; i0 < MQ; i0 += 8) {
        float v[8], u[8], rv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = u[i] = 0.f, rv[i] = resid(m0 + i0 + i);
        for (int cc = 0; cc < cnt; ++cc) {
          const float* pc = p0 + (size_t)cc * slot;
          float t[8], t2[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const bool in = m0 + i0 + i < M;
            t[i] = in ? __ldcg(pc + (size_t)(i0 + i) * NR * kQ4Rows) : 0.f;
            t2[i] = (NR == 2 && in) ? __ldcg(pc + (size_t)(i0 + i) * NR * kQ4Rows + kQ4Rows) : 0.f;
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) v[i] += t[i], u[i] += t2[i];
        }
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if (m0 + i0 + i < M && row < Nout) finish(m0 + i0 + i, v[i], u[i], rv[i]);
      }
      if (lane == 0) counters[b * DW + warp] = 0u;
    }
    q4_wait<0>();  // copies in flight land before the CTA leaves
  }
  tc_fence_before();
  __syncthreads();
  if (warp == DW + 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kQ4TmemCols) : "memory");
  }
}

// ---------------------------------------------------------------- host side
static int q4_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        n <= 0)
      n = 152;
  }
  return n;
}

static int q4_mt(int M) { return M <= 32 ? 32 : 64; }
static int q4_v(int groups) { return groups % 8 == 0 ? 8 : groups % 4 == 0 ? 4 : groups % 2 == 0 ? 2 : 1; }

bool q4tc_ok(int wquant, int epi, int M, int N, int K) {
  if ((wquant != FP_W_INT4_G128 && wquant != FP_W_INT8) || M < 17 || M > 64 || N < 1 || K < 128 || K % 128 != 0)
    return false;
  if (epi == FP_EPI_SWIGLU && N % 2 != 0) return false;
  const long long nout = epi == FP_EPI_SWIGLU ? N / 2 : N;
  const long long blocks = (nout + kQ4Rows - 1) / kQ4Rows;
  return blocks * kQ4DeqWarps <= kLinTicketSlots && tensor_maps_available();
}

// int4 always; int8 beyond 32 tokens or for long rows.  Measured at the
// 70B-shaped block's linears, microseconds on tcgen05 against mma.sync: 32
// tokens QKV 45.3 / 41.0, O 39.3 / 35.8, gate+up 173.9 / 165.4, down (K
// 28672) 86.2 / 118.9; 64 tokens 48.8 / 81.3, 45.1 / 70.3, 180.3 / 267.1,
// 96.0 / 204.7.  An int8 item carries half the weights of an int4 item for
// the same hand-offs, while the mma.sync GEMV's cost grows with the tokens.
bool q4tc_preferred(int wquant, int M, int K) { return wquant != FP_W_INT8 || M > 32 || K >= 16384; }

size_t q4tc_ws_bytes(int epi, int M, int N, int K) {
  const int nr = epi == FP_EPI_SWIGLU ? 2 : 1;
  const long long nout = nr == 2 ? N / 2 : N;
  const long long blocks = (nout + kQ4Rows - 1) / kQ4Rows;
  const long long ctas = std::min<long long>(blocks * (K / 64), q4_sms());  // items are at least 64 k
  return (size_t)kLinTicketSlots * 4 + (size_t)(blocks + ctas) * M * nr * kQ4Rows * 4;
}

template <int MT, int EPI, int WQ, int KI>
static cudaError_t launch_q4_t(const uint8_t* codes, const CUtensorMap& mx, int M, int N, int K,
                               const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* Y, void* ws,
                               int32_t* err, cudaStream_t s) {
  constexpr int NR = EPI == FP_EPI_SWIGLU ? 2 : 1;
  auto kern = gemv_q4tc_kernel<MT, EPI, WQ, KI>;
  const int smem = std::max(Q4Geom<MT, NR, WQ, KI>::kSmem, kQ4MinSmem);
  static std::atomic<unsigned long long> attr{0};
  FP_CUDA_TRY(smem_limit_once(kern, smem, &attr));
  const int nout = NR == 2 ? N / 2 : N;
  const long long blocks = (nout + kQ4Rows - 1) / kQ4Rows;
  const int S = K / 128;
  const long long total = blocks * (K / KI);  // items
  const int ctas = (int)std::min<long long>(total, q4_sms());
  unsigned* counters = (unsigned*)ws;
  float* part = (float*)((char*)ws + (size_t)kLinTicketSlots * 4);
  return launch(kern, dim3(ctas), dim3(kQ4Threads), (size_t)smem, s, mx, codes, M, N, scales, zeros, R, Y, total, S,
                WQ == FP_W_INT4_G128 ? q4_v(S) : 1, part, counters, err);
}

// k per item: int4 two groups where K allows (SwiGLU items already carry two
// matrices' groups), else one; int8 128, with SwiGLU 64 of each matrix
template <int MT, int WQ>
static cudaError_t launch_q4_w(int epi, const uint8_t* mw, const CUtensorMap& mx, int M, int N, int K,
                               const uint16_t* scales, const uint16_t* zeros, const uint16_t* R, void* Y, void* ws,
                               int32_t* err, cudaStream_t s) {
  constexpr bool I4 = WQ == FP_W_INT4_G128;
  constexpr int K2 = I4 ? 256 : 128;  // the larger item
  const bool two = I4 && (K / 128) % 2 == 0;
  switch (epi) {
    case FP_EPI_STORE:
      return two ? launch_q4_t<MT, FP_EPI_STORE, WQ, K2>(mw, mx, M, N, K, scales, zeros, R, Y, ws, err, s)
                 : launch_q4_t<MT, FP_EPI_STORE, WQ, 128>(mw, mx, M, N, K, scales, zeros, R, Y, ws, err, s);
    case FP_EPI_RESID:
      return two ? launch_q4_t<MT, FP_EPI_RESID, WQ, K2>(mw, mx, M, N, K, scales, zeros, R, Y, ws, err, s)
                 : launch_q4_t<MT, FP_EPI_RESID, WQ, 128>(mw, mx, M, N, K, scales, zeros, R, Y, ws, err, s);
    case FP_EPI_SWIGLU:
      return launch_q4_t<MT, FP_EPI_SWIGLU, WQ, I4 ? 128 : 64>(mw, mx, M, N, K, scales, zeros, R, Y, ws, err, s);
    default:
      return two ? launch_q4_t<MT, FP_EPI_F32, WQ, K2>(mw, mx, M, N, K, scales, zeros, R, Y, ws, err, s)
                 : launch_q4_t<MT, FP_EPI_F32, WQ, 128>(mw, mx, M, N, K, scales, zeros, R, Y, ws, err, s);
  }
}

cudaError_t launch_q4tc(int wquant, int epi, const uint16_t* x, int M, int N, int K, const void* codes,
                        const uint16_t* scales, const uint16_t* zeros, const uint16_t* residual, void* y, void* ws,
                        size_t ws_bytes, int32_t* err, cudaStream_t s) {
  if (!q4tc_ok(wquant, epi, M, N, K)) return cudaErrorInvalidValue;
  if (!ws || ws_bytes < q4tc_ws_bytes(epi, M, N, K)) return cudaErrorInvalidValue;
  CUtensorMap mx;
  const int mt = q4_mt(M);
  const uint8_t* mw = (const uint8_t*)codes;
  // x [M][K] bf16, box [mt rows][64]
  if (!make_tensor_map(&mx, x, M, K, 2, mt, 64, 128)) return cudaErrorInvalidValue;
  const bool i8 = wquant == FP_W_INT8;
  switch (mt) {
    case 32:
      return i8 ? launch_q4_w<32, FP_W_INT8>(epi, mw, mx, M, N, K, scales, zeros, residual, y, ws, err, s)
                : launch_q4_w<32, FP_W_INT4_G128>(epi, mw, mx, M, N, K, scales, zeros, residual, y, ws, err, s);
    default:
      return i8 ? launch_q4_w<64, FP_W_INT8>(epi, mw, mx, M, N, K, scales, zeros, residual, y, ws, err, s)
                : launch_q4_w<64, FP_W_INT4_G128>(epi, mw, mx, M, N, K, scales, zeros, residual, y, ws, err, s);
  }
}

}  // namespace fpk
