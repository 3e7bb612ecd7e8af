// Prefill attention on the tcgen05 tensor cores: paged cache of bf16 or int8
// codes with per-(token, KV head) fp32 scales, head_dim 128.
//
// o = softmax(q K^T / sqrt(hd) + causal mask) V for the S query rows of one
// (sequence, head) against cache positions 0..S-1 (Sec. 5.1: the block's
// attention).  CTA = 128 query rows of one (b, h), key tiles of 128; two
// CTAs per SM (256 TMEM columns and 97 KiB of shared memory each), so one
// CTA's softmax overlaps the other's MMAs and loads:
//   warp 0      TMA: the Q tile once (two 64-column boxes of the q rows), then
//               (bf16 cache) per key tile its K rows and its V rows page by
//               page (a [16][64] box per 16-token page and half of head_dim,
//               128-byte swizzle, one box per lane); K(t + 1) loads once S(t)
//               has read K(t), V(t + 1) once P(t) V(t) has read V(t);
//   warp 1      allocates the TMEM and issues the MMAs: S = Q K^T (M 128
//               queries, N 128 keys, K 16 over head_dim; K-major operands),
//               then O += P V (A = P from TMEM, B = V read MN-major);
//   warps 2-5   softmax, one query row (TMEM lane) per thread, over 32-column
//               chunks: a first pass for the row maximum (log2 domain), a
//               second for P = 2^(s - m) written as bf16 over the scores
//               already read.  The reference maximum m only moves when a tile
//               raises it by more than 2^8 (O and the row sum are rescaled
//               then); P never exceeds 256, and o / l is exact either way.
//   int8 cache: both products run on fp16 operands.  Warps 0, 6 and 7
//               (after warp 0 has issued the Q copy) convert the Q tile to
//               fp16 in place once, then widen the codes: each loads its
//               rows' 16-byte code chunks and turns each pair into the fp16
//               pair (1024 + q + 128) by one byte permute, minus 1152 --
//               exact -- in the same swizzled layout the TMA writes, and
//               stages the tile's K scales and its V scales times 2^sigma;
//               the softmax multiplies each score column by its K scale and
//               each P column by its scaled V scale in fp32 (the row sum
//               takes the unscaled P) and packs P as fp16.  sigma, one per
//               CTA, is the largest power of two keeping 256 * (largest V
//               scale of the sequence) * 2^sigma within 65280, so P stays in
//               the fp16 normal range; the output divides it out.  A q beyond
//               the fp16 range sets status 3.
// TMEM columns: scores S [0, 128) with P over [0, 64), O [128, 256).  Every
// mbarrier wait is bounded (error 2 past the limit); a page id out of range
// reads zeros and sets error 1.
#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace fpk {

constexpr int kPaB = 128;  // query rows per CTA = keys per tile
constexpr int kPaHD = 128;
constexpr int kPaWiden = 3;                                 // int8 cache: warps widening codes (0, 6, 7)
constexpr int kPaWRows = (kPaB + 4 * kPaWiden - 1) / (4 * kPaWiden);  // tile rows per widening thread
template <bool KV8>
constexpr int pa_threads() { return KV8 ? 256 : 192; }
constexpr uint32_t kPaTmemCols = 256;
constexpr uint32_t kPaS = 0, kPaO = 128;
constexpr int kPaHalf = kPaB * 128;          // bytes of one [128 rows][64 bf16] swizzled half
constexpr int kPaTile = 2 * kPaHalf;         // one [128][128] bf16 operand
constexpr int kPaSmem = 3 * kPaTile + 1024;  // Q, K, V, alignment
constexpr float kPaLog2e = 1.4426950408889634f;
// score columns per TMEM load in the softmax (64-column loads measured
// slower: 201 / 319 against 211 / 356 TFLOP/s at the 7B / 13B shapes)
constexpr int kPaCW = 32;
constexpr float kPaSlack = 8.f;  // log2 of the largest P allowed before the reference maximum moves

// Shared-memory descriptor of an MN-major operand with 128-byte swizzle:
// 64-element atoms along MN `lbo` bytes apart, 8-row groups along K 1024
// bytes apart.
FP_DEV uint64_t sdesc_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// 16 consecutive 32-bit columns into this thread's TMEM lane.
FP_DEV void pa_st16(uint32_t taddr, const uint32_t* r) { tc_st16(taddr, r); }

// 2^x by the hardware approximation (subnormal results flush to zero: P
// values below 2^-126 carry no weight next to the row's maximum of 1 .. 256).
FP_DEV float pa_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// (lo, hi) -> bf16x2, round to nearest even.
FP_DEV uint32_t pa_pack(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// (lo, hi) -> fp16x2, round to nearest even.
FP_DEV uint32_t pa_pack_h(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Signed bytes a and b of w as the fp16 pair (q_a, q_b), exact: the byte
// permute places q + 128 under the fp16 exponent of 1024 (0x64nn = 1024 + nn),
// one fp16x2 subtraction of 1152 leaves q.
FP_DEV uint32_t pa_i8h2(uint32_t u, uint32_t sel) {
  uint32_t h = __byte_perm(u, 0x64646464u, sel);
  asm("sub.rn.f16x2 %0, %0, %1;" : "+r"(h) : "r"(0x64806480u));
  return h;
}

template <bool KV8>
__global__ void __launch_bounds__(pa_threads<KV8>(), 2)
    attn_prefill_tc_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                           const __grid_constant__ CUtensorMap map_v, const int8_t* __restrict__ k8,
                           const int8_t* __restrict__ v8, const float* __restrict__ k_scale,
                           const float* __restrict__ v_scale, int S, int H, int Hkv, int page_size,
                           const int32_t* __restrict__ page_table, int pages_per_seq, int n_pages,
                           uint16_t* __restrict__ out, int32_t* err) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t qfull, qconv, kfull, kempty, vfull, vempty, sfull, pfull, ofull, mma_done;
  __shared__ float s_vmax[KV8 ? 3 : 1];  // int8: the widening warps' largest V scales
  __shared__ float s_unscale;             // int8: 2^-sigma, removed from the output
  __shared__ uint32_t tmem_base;
  __shared__ int abort_word;
  __shared__ __align__(16) float s_scl[KV8 ? 4 * kPaB : 4];  // int8: [K, V][tile parity][key] scales
  volatile int* abort_flag = &abort_word;
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  uint8_t* sK = smem + kPaTile;
  uint8_t* sV = smem + 2 * kPaTile;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int kvh = h / (H / Hkv);
  const int q0 = qt * kPaB;
  const int nt = (min(q0 + kPaB, S) - 1) / kPaB + 1;  // key tiles up to the diagonal
  auto fail = [&]() {
    *abort_flag = 1;
    if (err) atomicExch(err, 2);
  };

  pdl_trigger();
  if (threadIdx.x == 0) {
    mbar_init(&qfull, 1);
    mbar_init(&qconv, kPaWiden);  // int8: the widening warps converted Q to fp16
    mbar_init(&kfull, KV8 ? kPaWiden : 1);
    mbar_init(&kempty, 1);
    mbar_init(&vfull, KV8 ? kPaWiden : 1);
    mbar_init(&vempty, 1);
    mbar_init(&sfull, 1);
    mbar_init(&pfull, 4);
    mbar_init(&ofull, 1);
    mbar_init(&mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                 "r"(kPaTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  pdl_wait();

  if (KV8 && (warp == 0 || warp >= 6)) {
    // ---------------- int8 cache: the Q copy, then widening of the key tiles
    if (warp == 0 && lane == 0) {
      mbar_expect_tx(&qfull, kPaTile);
      tma_load_2d(sQ, &map_q, h * kPaHD, b * S + q0, &qfull);
      tma_load_2d(sQ + kPaHalf, &map_q, h * kPaHD + 64, b * S + q0, &qfull);
    }
    const int wi = (warp == 0 ? 0 : warp - 5) * 32 + lane;  // 0 .. 95
    const int c = wi & 7;                                     // code chunk: head_dim 16c .. 16c + 15
    const int rbase = wi >> 3;                                // tile rows rbase + 12i (< 128)
    const int32_t* ptv = page_table + (long long)b * pages_per_seq;
    // sigma: from the largest V scale over the keys this CTA reads
    float vmax = 0.f;
    const int nkeys = min(q0 + kPaB, S);
    for (int key = wi; key < nkeys; key += 32 * kPaWiden) {
      const int pg = __ldg(ptv + key / page_size);
      if (pg >= 0 && pg < n_pages) vmax = fmaxf(vmax, __ldg(v_scale + (pg * Hkv + kvh) * page_size + key % page_size));
    }
    vmax = warp_max(vmax);
    if (lane == 0) s_vmax[warp == 0 ? 0 : warp - 5] = vmax;
    asm volatile("bar.sync 1, %0;" ::"n"(32 * kPaWiden) : "memory");
    vmax = fmaxf(fmaxf(s_vmax[0], s_vmax[1]), s_vmax[2]);
    // 2^sigma with 256 * vmax * 2^sigma <= 65280 (vmax = 0: no V weight at all)
    const int sigma = vmax > 0.f ? min(60, max(-60, (int)floorf(log2f(255.f / vmax)))) : 0;
    const float vmul = exp2f((float)sigma);
    // published before the first code tile, which every softmax wait follows
    if (wi == 0) s_unscale = exp2f((float)-sigma);
    // Q to fp16 in place (the element order of the swizzled tile is kept)
    bool ok = __all_sync(0xffffffffu, mbar_wait(&qfull, 0));
    if (ok) {
      bool over = false;
      for (int i = wi; i < kPaTile / 16; i += 32 * kPaWiden) {
        uint4* p = reinterpret_cast<uint4*>(sQ) + i;
        const uint4 v = *p;
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
        uint32_t o[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 f = bf2x2f(w4[j]);
          over |= fabsf(f.x) > 65504.f || fabsf(f.y) > 65504.f;
          o[j] = pa_pack_h(f.x, f.y);
        }
        *p = make_uint4(o[0], o[1], o[2], o[3]);
      }
      if (over && err) atomicExch(err, 3);  // q outside the fp16 range: the output is invalid
      fence_proxy_async();
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&qconv);
    // its bf16 form is chunks cb, cb + 1 of half c / 4 of the swizzled row;
    // the lanes of the upper half store the odd chunk first, so the eight
    // lanes of one row write eight distinct 16-byte bank groups
    const int cb = 2 * (c & 3), half_off = (c >> 2) * kPaHalf;
    const int32_t* pt = ptv;
    for (int t = 0; t < nt && ok; ++t) {
      int rowi[kPaWRows];  // pool row of each of the thread's keys (< 2^31); -1 reads zeros
#pragma unroll
      for (int i = 0; i < kPaWRows; ++i) {
        const int row = rbase + 4 * kPaWiden * i, key = t * kPaB + row;
        rowi[i] = -1;
        if (row < kPaB && key < S) {
          const int pg = __ldg(pt + key / page_size);
          if (pg >= 0 && pg < n_pages) rowi[i] = (pg * Hkv + kvh) * page_size + key % page_size;
          else if (err && c == 0) atomicExch(err, 1);
        }
      }
      // the tile's K and V scales go out with its K codes: the softmax reads
      // both once S(t) is complete, which only the K tile's barrier precedes
      float sck[kPaWRows], scv[kPaWRows];
#pragma unroll
      for (int i = 0; i < kPaWRows; ++i) {
        sck[i] = (c == 0 && rowi[i] >= 0) ? __ldg(k_scale + rowi[i]) : 0.f;
        scv[i] = (c == 0 && rowi[i] >= 0) ? __ldg(v_scale + rowi[i]) * vmul : 0.f;
      }
#pragma unroll 1
      for (int which = 0; which < 2; ++which) {
        const int8_t* pool = which ? v8 : k8;
        uint4 w[kPaWRows];
        // the codes are read before the wait for the buffer
#pragma unroll
        for (int i = 0; i < kPaWRows; ++i)
          w[i] = rowi[i] >= 0 ? ld_nc16(pool + (long long)rowi[i] * kPaHD + c * 16) : make_uint4(0, 0, 0, 0);
        ok = t == 0 || mbar_wait(which ? &vempty : &kempty, (t - 1) & 1);
        if (!__all_sync(0xffffffffu, ok) || __any_sync(0xffffffffu, *abort_flag != 0)) {
          ok = false;
          break;
        }
        uint8_t* dst = (which ? sV : sK) + half_off;
#pragma unroll
        for (int i = 0; i < kPaWRows; ++i) {
          const int row = rbase + 4 * kPaWiden * i, sw = row & 7;
          if (row >= kPaB) break;
          const uint32_t ww[4] = {w[i].x ^ 0x80808080u, w[i].y ^ 0x80808080u, w[i].z ^ 0x80808080u,
                                  w[i].w ^ 0x80808080u};
          uint32_t o[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) o[j] = pa_i8h2(ww[j >> 1], (j & 1) ? 0x4342 : 0x4140);
          const uint4 e = make_uint4(o[0], o[1], o[2], o[3]), f = make_uint4(o[4], o[5], o[6], o[7]);
          uint8_t* rp = dst + row * 128;
          if (c < 4) {
            *reinterpret_cast<uint4*>(rp + ((cb ^ sw) << 4)) = e;
            *reinterpret_cast<uint4*>(rp + (((cb + 1) ^ sw) << 4)) = f;
          } else {
            *reinterpret_cast<uint4*>(rp + (((cb + 1) ^ sw) << 4)) = f;
            *reinterpret_cast<uint4*>(rp + ((cb ^ sw) << 4)) = e;
          }
          if (which == 0 && c == 0) {
            // buffer t & 1 was last read by the softmax of tile t - 2, which
            // completed before S(t - 1) was issued and so before this K tile's wait
            s_scl[(t & 1) * kPaB + row] = sck[i];
            s_scl[(2 + (t & 1)) * kPaB + row] = scv[i];
          }
        }
        fence_proxy_async();  // the MMAs read the tile through the async proxy
        __syncwarp();
        if (lane == 0) mbar_arrive(which ? &vfull : &kfull);
      }
    }
    if (!ok && lane == 0) fail();
  } else if (warp == 0) {
    // ---------------- TMA producer: lanes 0-15 each copy one [16][64] box of
    // a key tile (page lane & 7, head_dim half lane >> 3); lane 0 arms the
    // barriers.  The next tile's page ids are read while this one is in flight.
    const int32_t* pt = page_table + (long long)b * pages_per_seq;
    const int pg = lane & 7, half = (lane >> 3) & 1;
    auto page_row = [&](int t) {  // pool row of this lane's page of tile t; -16 reads zeros
      const int key0 = t * kPaB + pg * 16;
      if (lane >= 16 || key0 >= S) return -16;
      const int id = __ldg(pt + key0 / page_size);
      if (id >= 0 && id < n_pages) return (id * Hkv + kvh) * page_size;
      if (err && half == 0) atomicExch(err, 1);
      return -16;
    };
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(&map_k) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(&map_v) : "memory");
      mbar_expect_tx(&qfull, kPaTile);
      tma_load_2d(sQ, &map_q, h * kPaHD, b * S + q0, &qfull);
      tma_load_2d(sQ + kPaHalf, &map_q, h * kPaHD + 64, b * S + q0, &qfull);
    }
    int row = page_row(0);
    int kiss = 0, viss = 0;
    bool ok = true;
    for (int t = 0; t < nt; ++t) {
      if (t > 0) {
        ok = mbar_wait(&kempty, (t - 1) & 1);
        if (!__all_sync(0xffffffffu, ok) || __any_sync(0xffffffffu, *abort_flag != 0)) {
          ok = false;
          break;
        }
      }
      if (lane == 0) mbar_expect_tx(&kfull, kPaTile);
      __syncwarp();
      if (lane < 16) tma_load_2d(sK + half * kPaHalf + pg * 2048, &map_k, half * 64, row, &kfull);
      kiss = t + 1;
      if (t > 0) {
        ok = mbar_wait(&vempty, (t - 1) & 1);
        if (!__all_sync(0xffffffffu, ok) || __any_sync(0xffffffffu, *abort_flag != 0)) {
          ok = false;
          break;
        }
      }
      if (lane == 0) mbar_expect_tx(&vfull, kPaTile);
      __syncwarp();
      if (lane < 16) tma_load_2d(sV + half * kPaHalf + pg * 2048, &map_v, half * 64, row, &vfull);
      viss = t + 1;
      if (t + 1 < nt) row = page_row(t + 1);
    }
    if (lane == 0) {
      if (!ok) fail();
      // copies still in flight land before the CTA leaves
      mbar_wait(&qfull, 0);
      if (kiss > 0) mbar_wait(&kfull, (kiss - 1) & 1);
      if (viss > 0) mbar_wait(&vfull, (viss - 1) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      // Q, K both K-major; V MN-major.  int8 cache: fp16 operands (A and B
      // of one MMA always share their type), bf16 cache: bf16
      constexpr uint32_t f16 = KV8 ? ((1u << 7) | (1u << 10)) : 0u;
      constexpr uint32_t idesc_s = tc_idesc(kPaB, kPaB) & ~f16;
      constexpr uint32_t idesc_o = (tc_idesc(kPaB, kPaHD) | (1u << 16)) & ~f16;
      bool ok = KV8 ? mbar_wait(&qconv, 0) : mbar_wait(&qfull, 0);
      const uint32_t q = smem_u32(sQ), k = smem_u32(sK), v = smem_u32(sV);
      for (int t = 0; t < nt && ok; ++t) {
        // S(t) overwrites P(t - 1): its P V has completed (in order with this thread's MMAs)
        ok = mbar_wait(&kfull, t & 1) && (t == 0 || mbar_wait(&ofull, (t - 1) & 1)) && !*abort_flag;
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kPaHD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPaHalf + (kk & 3) * 32;
          tc_mma(tmem + kPaS, sdesc(q + off), sdesc(k + off), idesc_s, kk > 0 ? 1u : 0u);
        }
        tc_commit(&sfull);
        tc_commit(&kempty);
        ok = mbar_wait(&pfull, t & 1) && mbar_wait(&vfull, t & 1) && !*abort_flag;
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kPaB / 16; ++kk)  // 16 keys: two 8-row groups of the V tile
          tc_mma_ts(tmem + kPaO, tmem + kPaS + kk * 8, sdesc_mn(v + kk * 2048, kPaHalf), idesc_o,
                    (t > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&ofull);
        tc_commit(&vempty);
      }
      if (!ok) fail();
      tc_commit(&mma_done);
      mbar_wait(&mma_done, 0);
    }
  } else {
    // ---------------- softmax: thread = query row (TMEM lane 32 (warp % 4) + lane)
    const int quad = warp & 3, row = quad * 32 + lane;
    const int qrow = q0 + row;  // position in the sequence
    const uint32_t lane_base = tmem + ((uint32_t)(quad * 32) << 16);
    const float scale = kPaLog2e * rsqrtf((float)kPaHD);
    float m = -INFINITY, l = 0.f;  // reference maximum (log2 domain) and row sum
    bool ok = true;
    for (int t = 0; t < nt; ++t) {
      ok = mbar_wait(&sfull, t & 1);
      if (!__all_sync(0xffffffffu, ok) || __any_sync(0xffffffffu, *abort_flag != 0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int key0 = t * kPaB;
      // keys past this row or past S only occur in the diagonal tile
      const bool masked = key0 + kPaB - 1 > q0 || key0 + kPaB > S;
      // raw scores of chunk c (kPaCW columns); masked keys read -inf
      auto load_raw = [&](auto mask, int c, float* v) {
        uint32_t r[kPaCW];
        tc_ld<kPaCW>(lane_base + kPaS + c * kPaCW, r);
        if constexpr (KV8) {
          // K scale of each key column (masked columns are overwritten below)
          const float4* k4 = reinterpret_cast<const float4*>(s_scl + (t & 1) * kPaB + c * kPaCW);
#pragma unroll
          for (int i = 0; i < kPaCW / 4; ++i) {
            const float4 f = k4[i];
            r[4 * i] = __float_as_uint(__uint_as_float(r[4 * i]) * f.x);
            r[4 * i + 1] = __float_as_uint(__uint_as_float(r[4 * i + 1]) * f.y);
            r[4 * i + 2] = __float_as_uint(__uint_as_float(r[4 * i + 2]) * f.z);
            r[4 * i + 3] = __float_as_uint(__uint_as_float(r[4 * i + 3]) * f.w);
          }
        }
#pragma unroll
        for (int i = 0; i < kPaCW; ++i) {
          v[i] = __uint_as_float(r[i]);
          if constexpr (decltype(mask)::value) {
            const int key = key0 + c * kPaCW + i;
            if (key > qrow || key >= S) v[i] = -INFINITY;
          }
        }
      };
      // pass 1: the row maximum of the raw scores (scale > 0 keeps the order)
      auto row_max = [&](auto mask) {
        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll 1
        for (int c = 0; c < kPaB / kPaCW; ++c) {
          float v[kPaCW];
          load_raw(mask, c, v);
#pragma unroll
          for (int i = 0; i < kPaCW; ++i) m4[i & 3] = fmaxf(m4[i & 3], v[i]);
        }
        return fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
      };
      const float mraw = masked ? row_max(std::true_type{}) : row_max(std::false_type{});
      const float mx = mraw * scale;
      // move the reference when the tile would exceed it by more than 2^kPaSlack
      float corr = 1.f;
      if (mx > m + kPaSlack) {
        corr = exp2f(m - mx);  // 0 on the first tile
        m = mx;
        l *= corr;
      }
      if (t > 0 && __any_sync(0xffffffffu, corr != 1.f)) {
        // O holds P V of the earlier tiles (complete: S(t) was issued after it)
#pragma unroll 1
        for (int c = 0; c < kPaHD / 32; ++c) {
          uint32_t r[32];
          tc_ld<32>(lane_base + kPaO + c * 32, r);
#pragma unroll
          for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * corr);
          tc_st32(lane_base + kPaO + c * 32, r);
        }
      }
      // pass 2: P = 2^(s scale - m) as bf16 pairs over the score columns already read
      const float mref = m == -INFINITY ? 0.f : m;
      auto write_p = [&](auto mask) {
        float p4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
        for (int c = 0; c < kPaB / kPaCW; ++c) {
          float v[kPaCW];
          load_raw(mask, c, v);
          uint32_t pw[kPaCW / 2];
#pragma unroll
          for (int i = 0; i < kPaCW; i += 2) {
            const float p0 = pa_ex2(fmaf(v[i], scale, -mref)), p1 = pa_ex2(fmaf(v[i + 1], scale, -mref));
            p4[i & 3] += p0;
            p4[(i + 1) & 3] += p1;
            if constexpr (KV8) {
              // V scale of each key column: P V then takes the codes as they are
              const float2 vs = *reinterpret_cast<const float2*>(s_scl + (2 + (t & 1)) * kPaB + c * kPaCW + i);
              pw[i / 2] = pa_pack_h(p0 * vs.x, p1 * vs.y);
            } else {
              pw[i / 2] = pa_pack(p0, p1);
            }
          }
          pa_st16(lane_base + kPaS + c * (kPaCW / 2), pw);
        }
        return (p4[0] + p4[1]) + (p4[2] + p4[3]);
      };
      const float ps = masked ? write_p(std::true_type{}) : write_p(std::false_type{});
      l += ps;
      tc_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pfull);
    }
    if (ok) {
      ok = mbar_wait(&ofull, (nt - 1) & 1);
      ok = __all_sync(0xffffffffu, ok);
    }
    if (ok) {
      tc_fence_after();
      // int8 cache: P carried the V scales times 2^sigma
      const float inv = (KV8 ? s_unscale : 1.f) / l;
      uint16_t* dst = out + ((long long)b * S + qrow) * ((long long)H * kPaHD) + (long long)h * kPaHD;
#pragma unroll 1
      for (int c = 0; c < kPaHD / 32; ++c) {
        uint32_t r[32];
        tc_ld<32>(lane_base + kPaO + c * 32, r);
        if (qrow < S) {
#pragma unroll
          for (int i = 0; i < 32; i += 8)
            *reinterpret_cast<uint4*>(dst + c * 32 + i) =
                make_uint4(pack_bf2(__uint_as_float(r[i]) * inv, __uint_as_float(r[i + 1]) * inv),
                           pack_bf2(__uint_as_float(r[i + 2]) * inv, __uint_as_float(r[i + 3]) * inv),
                           pack_bf2(__uint_as_float(r[i + 4]) * inv, __uint_as_float(r[i + 5]) * inv),
                           pack_bf2(__uint_as_float(r[i + 6]) * inv, __uint_as_float(r[i + 7]) * inv));
        }
      }
    } else if (lane == 0) {
      fail();
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kPaTmemCols) : "memory");
  }
}

bool attention_prefill_tc_ok(int B, int S, int n_heads, const fp_kv_view& kv, const void* q, int q_stride) {
  const bool kv8 = kv.kvquant == FP_KV_INT8;
  return (kv.kvquant == FP_KV_BF16 || (kv8 && kv.k_scale && kv.v_scale)) && kv.head_dim == kPaHD &&
         kv.page_size == 16 && B >= 1 && S >= 1 && n_heads % kv.n_kv_heads == 0 && q_stride % 8 == 0 &&
         ((uintptr_t)q & 15) == 0 && ((uintptr_t)kv.k_pool & 15) == 0 && ((uintptr_t)kv.v_pool & 15) == 0 &&
         (long long)kv.n_pages * kv.n_kv_heads * kv.page_size < (1LL << 31) && tensor_maps_available();
}

template <bool KV8>
static cudaError_t launch_pa_tc(const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mv, int B, int S,
                                int n_heads, const fp_kv_view& kv, uint16_t* out, int32_t* err, cudaStream_t s) {
  static std::atomic<unsigned long long> attr{0};
  FP_CUDA_TRY(smem_limit_once(attn_prefill_tc_kernel<KV8>, kPaSmem, &attr));
  const dim3 grid((S + kPaB - 1) / kPaB, n_heads, B);
  return launch(attn_prefill_tc_kernel<KV8>, grid, dim3(pa_threads<KV8>()), (size_t)kPaSmem, s, mq, mk, mv,
                (const int8_t*)kv.k_pool, (const int8_t*)kv.v_pool, (const float*)kv.k_scale,
                (const float*)kv.v_scale, S, n_heads, kv.n_kv_heads, kv.page_size, kv.page_table, kv.pages_per_seq,
                kv.n_pages, out, err);
}

cudaError_t launch_attention_prefill_tc(const uint16_t* q, int q_stride, int B, int S, int n_heads,
                                        const fp_kv_view& kv, uint16_t* out, int32_t* err, cudaStream_t s) {
  CUtensorMap mq, mk, mv;
  const long long pool_rows = (long long)kv.n_pages * kv.n_kv_heads * kv.page_size;
  // q [B S][q_stride] bf16, box [128 rows][64]
  if (!make_tensor_map(&mq, q, (long long)B * S, q_stride, 2, kPaB, 64, 128)) return cudaErrorInvalidValue;
  if (kv.kvquant == FP_KV_INT8) return launch_pa_tc<true>(mq, mq, mq, B, S, n_heads, kv, out, err, s);
  // bf16 pools [pages Hkv 16][128], box [16 rows][64]
  if (!make_tensor_map(&mk, kv.k_pool, pool_rows, kPaHD, 2, 16, 64, 128) ||
      !make_tensor_map(&mv, kv.v_pool, pool_rows, kPaHD, 2, 16, 64, 128))
    return cudaErrorInvalidValue;
  return launch_pa_tc<false>(mq, mk, mv, B, S, n_heads, kv, out, err, s);
}

}  // namespace fpk
