// Prefill attention on the tcgen05 tensor cores: bf16 paged cache, head_dim
// 128.
//
// o = softmax(q K^T / sqrt(hd) + causal mask) V for the S query rows of one
// (sequence, head) against cache positions 0..S-1 (Sec. 5.1: the block's
// attention).  CTA = 128 query rows of one (b, h), key tiles of 128:
//   warp 0      TMA: the Q tile once (two 64-column boxes of the q rows), then
//               each key tile's K and V rows page by page (a [16][64] box per
//               16-token page and half of head_dim, 128-byte swizzle) into a
//               two-stage ring (kvfull / kvempty);
//   warp 1      allocates 512 TMEM columns and issues the MMAs: S = Q K^T
//               (M 128 queries, N 128 keys, K 16 over head_dim; K-major
//               operands) into one of two score buffers, then O += P V
//               (A = P from TMEM, B = V read MN-major from the same tile);
//   warps 2-5   softmax, one query row (TMEM lane) per thread: the row's 128
//               scores (tcgen05.ld), scale and causal mask, running maximum in
//               the log2 domain, P = 2^(s - m) as bf16 into TMEM, the O rescale
//               when the maximum grows, and at the end o / l stored as bf16.
// TMEM columns: scores S0 [0, 128), S1 [128, 256), O [256, 384), P [384, 448).
// The scores of key tile t + 1 are computed while the softmax works on tile
// t.  Every mbarrier wait is bounded (error 2 past the limit); a page id out
// of range reads zeros and sets error 1.
#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace fpk {

constexpr int kPaB = 128;  // query rows per CTA = keys per tile
constexpr int kPaHD = 128;
constexpr int kPaThreads = 192;
constexpr uint32_t kPaTmemCols = 512;
constexpr uint32_t kPaS0 = 0, kPaO = 256, kPaP = 384;
constexpr int kPaHalf = kPaB * 128;          // bytes of one [128 rows][64 bf16] swizzled half
constexpr int kPaTile = 2 * kPaHalf;         // one [128][128] bf16 operand
constexpr int kPaSmem = kPaTile + 2 * 2 * kPaTile + 1024;  // Q, two stages of K and V, alignment
constexpr float kPaLog2e = 1.4426950408889634f;

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

__global__ void __launch_bounds__(kPaThreads, 1)
    attn_prefill_tc_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                           const __grid_constant__ CUtensorMap map_v, int S, int H, int Hkv, int page_size,
                           const int32_t* __restrict__ page_table, int pages_per_seq, int n_pages,
                           uint16_t* __restrict__ out, int32_t* err) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t qfull, kvfull[2], kvempty[2], sfull[2], sempty[2], pfull, ofull, mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_word;
  volatile int* abort_flag = &abort_word;
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  auto sK = [&](int st) { return smem + kPaTile + st * 2 * kPaTile; };
  auto sV = [&](int st) { return smem + kPaTile + st * 2 * kPaTile + kPaTile; };
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
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kvfull[i], 1);
      mbar_init(&kvempty[i], 1);
      mbar_init(&sfull[i], 1);
      mbar_init(&sempty[i], 4);
    }
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

  if (warp == 0) {
    // ---------------- TMA producer
    if (lane == 0) {
      mbar_expect_tx(&qfull, kPaTile);
      tma_load_2d(sQ, &map_q, h * kPaHD, b * S + q0, &qfull);
      tma_load_2d(sQ + kPaHalf, &map_q, h * kPaHD + 64, b * S + q0, &qfull);
      const int32_t* pt = page_table + (long long)b * pages_per_seq;
      int issued = 0;
      for (int t = 0; t < nt; ++t) {
        const int st = t & 1;
        if (t >= 2 && (!mbar_wait(&kvempty[st], ((t >> 1) & 1) ^ 1) || *abort_flag)) {
          fail();
          break;
        }
        mbar_expect_tx(&kvfull[st], 2 * kPaTile);
        for (int pg = 0; pg < kPaB / 16; ++pg) {
          const int key0 = t * kPaB + pg * 16;
          int row = -16;  // wholly outside the pool: the box reads zeros
          if (key0 < S) {
            const int page = pt[key0 / page_size];
            if (page >= 0 && page < n_pages) row = (page * Hkv + kvh) * page_size;
            else if (err) atomicExch(err, 1);
          }
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            tma_load_2d(sK(st) + half * kPaHalf + pg * 2048, &map_k, half * 64, row, &kvfull[st]);
            tma_load_2d(sV(st) + half * kPaHalf + pg * 2048, &map_v, half * 64, row, &kvfull[st]);
          }
        }
        issued = t + 1;
      }
      // copies still in flight land before the CTA leaves
      mbar_wait(&qfull, 0);
      for (int j = max(0, issued - 2); j < issued; ++j) mbar_wait(&kvfull[j & 1], (j >> 1) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = tc_idesc(kPaB, kPaB);             // Q, K both K-major
      constexpr uint32_t idesc_o = tc_idesc(kPaB, kPaHD) | (1u << 16);  // V MN-major
      bool ok = mbar_wait(&qfull, 0);
      auto issue_s = [&](int t) -> bool {
        const int st = t & 1, sb = t & 1;
        if (!mbar_wait(&kvfull[st], (t >> 1) & 1)) return false;
        if (t >= 2 && !mbar_wait(&sempty[sb], ((t >> 1) & 1) ^ 1)) return false;
        tc_fence_after();
        const uint32_t q = smem_u32(sQ), k = smem_u32(sK(st));
#pragma unroll
        for (int kk = 0; kk < kPaHD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPaHalf + (kk & 3) * 32;
          tc_mma(tmem + kPaS0 + sb * kPaB, sdesc(q + off), sdesc(k + off), idesc_s, kk > 0 ? 1u : 0u);
        }
        tc_commit(&sfull[sb]);
        return true;
      };
      ok = ok && !*abort_flag && issue_s(0);
      for (int t = 0; t < nt && ok; ++t) {
        if (t + 1 < nt && !(ok = issue_s(t + 1))) break;
        if (!(ok = mbar_wait(&pfull, t & 1)) || *abort_flag) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t v = smem_u32(sV(t & 1));
#pragma unroll
        for (int kk = 0; kk < kPaB / 16; ++kk)  // 16 keys: two 8-row groups of the V tile
          tc_mma_ts(tmem + kPaO, tmem + kPaP + kk * 8, sdesc_mn(v + kk * 2048, kPaHalf), idesc_o,
                    (t > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&ofull);
        tc_commit(&kvempty[t & 1]);
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
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int t = 0; t < nt; ++t) {
      const int sb = t & 1;
      ok = mbar_wait(&sfull[sb], (t >> 1) & 1);
      if (!__all_sync(0xffffffffu, ok) || __any_sync(0xffffffffu, *abort_flag != 0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[kPaB];
#pragma unroll
      for (int c = 0; c < kPaB / 32; ++c) {
        uint32_t r[32];
        tc_ld<32>(lane_base + kPaS0 + sb * kPaB + c * 32, r);
#pragma unroll
        for (int i = 0; i < 32; ++i) s[c * 32 + i] = __uint_as_float(r[i]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sempty[sb]);

      // scale, causal mask, running maximum (log2 domain)
      const int key0 = t * kPaB;
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < kPaB; ++j) {
        const int key = key0 + j;
        const float v = (key > qrow || key >= S) ? -INFINITY : s[j] * scale;
        s[j] = v;
        mx = fmaxf(mx, v);
      }
      const float mnew = fmaxf(m, mx);
      const float mref = mnew == -INFINITY ? 0.f : mnew;
      const float corr = exp2f(m - mref);  // 0 on the first tile
      float ps = 0.f;
      uint32_t pw[kPaB / 2];
#pragma unroll
      for (int j = 0; j < kPaB; j += 2) {
        const float p0 = exp2f(s[j] - mref), p1 = exp2f(s[j + 1] - mref);
        ps += p0 + p1;
        pw[j / 2] = pack_bf2(p0, p1);
      }
      l = l * corr + ps;
      m = mnew;

      if (t > 0) {
        // the previous P V has completed: its P columns are free and O is final for it
        ok = mbar_wait(&ofull, (t - 1) & 1);
        if (!__all_sync(0xffffffffu, ok) || __any_sync(0xffffffffu, *abort_flag != 0)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(0xffffffffu, corr != 1.f)) {  // rescale O (warp-wide TMEM access)
#pragma unroll 1
          for (int c = 0; c < kPaHD / 32; ++c) {
            uint32_t r[32];
            tc_ld<32>(lane_base + kPaO + c * 32, r);
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * corr);
            tc_st32(lane_base + kPaO + c * 32, r);
          }
        }
      }
      tc_st32(lane_base + kPaP, pw);
      tc_st32(lane_base + kPaP + 32, pw + 32);
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
      const float inv = 1.f / l;
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
  return kv.kvquant == FP_KV_BF16 && kv.head_dim == kPaHD && kv.page_size == 16 && B >= 1 && S >= 1 &&
         n_heads % kv.n_kv_heads == 0 && q_stride % 8 == 0 && ((uintptr_t)q & 15) == 0 &&
         ((uintptr_t)kv.k_pool & 15) == 0 && ((uintptr_t)kv.v_pool & 15) == 0 &&
         (long long)kv.n_pages * kv.n_kv_heads * kv.page_size < (1LL << 31) && tensor_maps_available();
}

cudaError_t launch_attention_prefill_tc(const uint16_t* q, int q_stride, int B, int S, int n_heads,
                                        const fp_kv_view& kv, uint16_t* out, int32_t* err, cudaStream_t s) {
  CUtensorMap mq, mk, mv;
  const long long pool_rows = (long long)kv.n_pages * kv.n_kv_heads * kv.page_size;
  // q [B S][q_stride] bf16, box [128 rows][64]; pools [pages Hkv 16][128] bf16, box [16 rows][64]
  if (!make_tensor_map(&mq, q, (long long)B * S, q_stride, 2, kPaB, 64, 128) ||
      !make_tensor_map(&mk, kv.k_pool, pool_rows, kPaHD, 2, 16, 64, 128) ||
      !make_tensor_map(&mv, kv.v_pool, pool_rows, kPaHD, 2, 16, 64, 128))
    return cudaErrorInvalidValue;
  static bool attr = false;
  if (!attr) {
    FP_CUDA_TRY(cudaFuncSetAttribute(attn_prefill_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kPaSmem));
    attr = true;
  }
  const dim3 grid((S + kPaB - 1) / kPaB, n_heads, B);
  return launch(attn_prefill_tc_kernel, grid, dim3(kPaThreads), (size_t)kPaSmem, s, mq, mk, mv, S, n_heads,
                kv.n_kv_heads, kv.page_size, kv.page_table, kv.pages_per_seq, kv.n_pages, out, err);
}

}  // namespace fpk
