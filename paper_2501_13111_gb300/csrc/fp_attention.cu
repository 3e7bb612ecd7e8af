// Attention over the paged KV cache: decode (one query row per sequence,
// split over the context, then combined) and prefill (causal, flash-style
// with bf16 tensor-core MMAs).
//
// softmax(q K^T / sqrt(hd)) V with query head j reading KV head j / (H/Hkv)
// ("softmax activations" among the fingerprint's components, Sec. 1 "Our
// work"; the KV cache makes every decode step cost the same, Sec. 5.3 before
// Eq. 1).  Both kernels read K and V back from the cache; with the int8 cache
// the per-token scales multiply the scores (K) and the probabilities (V), so
// codes enter the arithmetic exactly.
#include <algorithm>

#include <cuda_fp16.h>

#include "common.cuh"
#include "kernels.cuh"

namespace fpk {

static constexpr float kLog2e = 1.4426950408889634f;

// =====================================================================
// Decode: grid (B * Hkv, splits); one CTA handles the G = H / Hkv query
// heads of one KV head over one chunk of the context.  The chunk's K and V
// stream through a ring of 64-token tiles in shared memory (cp.async, two
// tiles in flight; rows padded so ldmatrix is conflict-free).  Each of the 4
// warps takes 16 tokens of a tile: scores S = Q K^T and O += P V run on the
// tensor cores (mma.sync m16n8k16, fp32 accumulation; the G query heads are
// rows of the A operand), with an online softmax in the log2 domain on the
// score fragments.  bf16 caches enter as they are (P in bf16); int8 codes
// are widened exactly to fp16 in shared memory (P in fp16) and their
// per-token scales applied in fp32 to the scores (K) and to P (V).  The 4
// warps are merged at the end; a second kernel merges the context splits.
// =====================================================================
constexpr int kDecTT = 64;  // tokens per tile

// Ring depth: 3 tiles (two in flight, 2 CTAs per SM with the bf16 cache) when
// the (sequence, KV head) pairs leave SMs with room, else 2 tiles (one in
// flight) so that 3 CTAs share an SM -- with pairs to spare, more resident
// warps beat a deeper ring.
struct DecodeGeom {
  int chunk;   // positions per split (multiple of kDecTT)
  int splits;  // ceil(max_len / chunk)
  int nb;      // ring depth
};

static int dec_sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        n <= 0)
      n = 152;
  }
  return n;
}

// Resident decode CTAs per SM assumed by the split geometry for a ring depth
// (the bf16 ring takes 104 KB at 3 tiles, 70 KB at 2).
constexpr int dec_occ(int nb) { return nb == 2 ? 3 : 2; }
static int dec_ring_depth(long long pairs) { return pairs >= 2LL * dec_sm_count() ? 2 : 3; }

// Split count: the candidates are the counts a whole number of tiles per
// split produces; each is scored as (waves of resident CTAs) x (tiles per
// split + one tile of fixed cost), and the cheapest wins (fewer splits on a
// tie).  At most 4 splits or 2 waves' worth per (sequence, KV head) pair,
// whichever is more (and at least the splits that keep a split within
// kDecMaxChunkTiles tiles), so the count never grows with n_kv_heads and the
// workspace sized for n_kv_heads = 1 covers every launch.
constexpr int kDecMaxChunkTiles = 256;  // a split covers at most 16384 positions (bounds its page-id stage)

static int dec_min_splits(int tiles) { return (tiles + kDecMaxChunkTiles - 1) / kDecMaxChunkTiles; }

static int dec_max_splits(long long pairs, int tiles) {
  const long long slots = (long long)dec_sm_count() * dec_occ(2);  // the larger occupancy bounds both depths
  const long long s = std::max<long long>(std::min(tiles, 4), std::min<long long>(tiles, 2 * slots / std::max<long long>(1, pairs)));
  return (int)std::max<long long>(std::max<long long>(s, 1), dec_min_splits(tiles));
}

// occ > 0: CTAs per SM of the kernel the geometry is for (the int8 page-streaming
// kernel: 4); occ 0: the mma.sync tile kernel, whose ring depth sets it.
static DecodeGeom decode_geom(int B, int n_kv_heads, int max_len, int occ = 0) {
  const long long pairs = (long long)B * n_kv_heads;
  const int nb = dec_ring_depth(pairs);
  const long long slots = (long long)dec_sm_count() * (occ > 0 ? occ : dec_occ(nb));
  const int tiles = std::max(1, (max_len + kDecTT - 1) / kDecTT);
  const int smax = std::min(dec_max_splits(pairs, tiles),
                            (int)std::max<long long>(std::min<long long>(tiles, 4), 2 * slots / std::max(1LL, pairs)));
  DecodeGeom best{tiles * kDecTT, 1, nb};
  double best_t = 1e30;
  for (int s = std::max(1, dec_min_splits(tiles)); s <= smax; ++s) {
    const int per = (tiles + s - 1) / s;
    const int splits = (tiles + per - 1) / per;
    const long long ctas = pairs * splits;
    const double t = (double)((ctas + slots - 1) / slots) * (per + 1);
    if (t < best_t) {
      best_t = t;
      best.chunk = per * kDecTT;
      best.splits = (max_len + best.chunk - 1) / best.chunk;
    }
  }
  return best;
}

// The int8 cache with head_dim 128 (16-byte aligned pools, 16-token pages)
// runs the page-streaming kernel.  It shares the tile kernel's split
// geometry: scoring its 4 CTAs per SM split the 70B-shaped context in two,
// which measured slower (42 us against 36 us; each warp's ring fill and the
// merge weigh more on half the pages, and the combine pass is added).
static bool dec_i8_shape(int kvquant, int head_dim, int page_size) {
  return kvquant == FP_KV_INT8 && head_dim == 128 && page_size == 16;
}
static DecodeGeom decode_geom_for(int B, int n_kv_heads, int head_dim, int kvquant, int page_size, int max_len) {
  (void)head_dim, (void)kvquant, (void)page_size;
  return decode_geom(B, n_kv_heads, max_len);
}

int attention_decode_launches(int B, int n_kv_heads, int head_dim, int kvquant, int max_len) {
  return decode_geom_for(B, n_kv_heads, head_dim, kvquant, 16, max_len).splits == 1 ? 1 : 2;
}

int attention_decode_splits(int B, int n_kv_heads, int head_dim, int kvquant, int max_len) {
  return decode_geom_for(B, n_kv_heads, head_dim, kvquant, 16, max_len).splits;
}

size_t attention_decode_ws_bytes(int B, int n_heads, int head_dim, int max_len) {
  const int tiles = std::max(1, (max_len + kDecTT - 1) / kDecTT);
  const size_t rows = (size_t)B * n_heads * dec_max_splits(B, tiles);
  return rows * (size_t)(head_dim + 2) * sizeof(float);
}

FP_DEV void dec_cp_async16(void* smem, const void* gmem) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s), "l"(gmem) : "memory");
}
FP_DEV void dec_cp_async4(void* smem, const void* gmem) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(s), "l"(gmem) : "memory");
}

template <bool F16>
FP_DEV void dec_mma(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  if constexpr (F16) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
  } else {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
  }
}

FP_DEV void dec_ldsm_x4(uint32_t* r, const void* p, bool trans) {
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  if (trans)
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(a));
  else
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(a));
}

// Two fp32 values as an MMA operand word: bf16 or fp16 pair.
template <bool F16>
FP_DEV uint32_t dec_pack(float a, float b) {
  if constexpr (F16) {
    const __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
  } else {
    return pack_bf2(a, b);
  }
}

// int8 codes (4 per word) -> two fp16 pairs, exactly: fp16(1024 + (q + 128)) - 1152.
FP_DEV uint2 dec_i8_to_f16x4(uint32_t w) {
  const uint32_t x = w ^ 0x80808080u;
  const uint32_t lo = __byte_perm(x, 0x64646464u, 0x5140), hi = __byte_perm(x, 0x64646464u, 0x5342);
  const __half2 off = __float2half2_rn(1152.f);
  const __half2 a = __hsub2(*reinterpret_cast<const __half2*>(&lo), off);
  const __half2 b = __hsub2(*reinterpret_cast<const __half2*>(&hi), off);
  return make_uint2(*reinterpret_cast<const uint32_t*>(&a), *reinterpret_cast<const uint32_t*>(&b));
}

template <int HD, int KVQ, int NB>
constexpr size_t dec_smem_bytes() {
  constexpr size_t ld = HD + 8;  // padded 16-bit row (elements)
  if (KVQ == FP_KV_BF16) return (size_t)NB * kDecTT * ld * 2 * 2;
  // int8: ring of code rows (HD + 16 bytes), per-token scales, one fp16 tile of K and V
  return (size_t)NB * kDecTT * (HD + 16) * 2 + (size_t)NB * kDecTT * 2 * sizeof(float) +
         (size_t)kDecTT * ld * 2 * 2;
}

// The ring, which also holds the 4-warp merge buffer after the loop; the
// chunk's page ids follow it.
template <int HD, int KVQ, int G, int NB>
constexpr size_t dec_stage_bytes() {
  return std::max(dec_smem_bytes<HD, KVQ, NB>(), (size_t)4 * G * (HD + 2) * sizeof(float));
}

// Workspace layout for (b, h, split): o [HD] fp32 (un-normalised, relative to
// m), then (m, l) in the log2 domain.
template <int HD, int KVQ, int G, int NB>
__global__ void __launch_bounds__(128) attn_decode_kernel(const uint16_t* __restrict__ q, int q_stride, int H,
                                                          fp_kv_view kv, const int32_t* __restrict__ len,
                                                          int len_add, int max_len, int chunk, int splits,
                                                          float* __restrict__ ws, uint16_t* __restrict__ out,
                                                          int32_t* err) {
  constexpr int TT = kDecTT, LD = HD + 8;
  constexpr bool I8 = KVQ == FP_KV_INT8;
  constexpr int RAWB = I8 ? HD + 16 : LD * 2;  // bytes per staged row
  constexpr int CPR = (I8 ? HD : HD * 2) / 16;  // 16-byte chunks per row
  constexpr int NT = HD / 8;                    // n8 tiles of the output
  static_assert(G <= 8, "query heads per KV head are rows 0..7 of the MMA tile");
  static_assert(TT == 4 * 16, "each of the 4 warps takes 16 tokens of a tile");
  extern __shared__ __align__(16) uint8_t smem[];
  uint8_t* sK = smem;                                          // [NB][TT][RAWB]
  uint8_t* sV = sK + NB * TT * RAWB;                           // [NB][TT][RAWB]
  float* sKs = reinterpret_cast<float*>(sV + NB * TT * RAWB);  // int8: [NB][TT]
  float* sVs = sKs + NB * TT;
  uint16_t* cK = reinterpret_cast<uint16_t*>(sVs + NB * TT);  // int8: fp16 [TT][LD]
  uint16_t* cV = cK + TT * LD;
  pdl_trigger();
  pdl_wait();
  const int Hkv = kv.n_kv_heads;
  const int b = blockIdx.x / Hkv, kvh = blockIdx.x % Hkv;
  const int split = blockIdx.y;
  int T = len[b] + len_add;
  if (T > max_len) {  // never past the positions the grid and the page table cover
    if (err && split == 0 && threadIdx.x == 0) atomicExch(err, 1);
    T = max_len;
  }
  const int t0 = split * chunk;
  if (t0 >= T) {
    if (splits == 1)  // empty context: zero output
      for (int i = threadIdx.x; i < G * HD; i += 128) out[((long long)b * H + kvh * G) * HD + i] = 0;
    return;
  }
  const int t1 = min(T, t0 + chunk);
  const int ntile = (t1 - t0 + TT - 1) / TT;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // ---- the page ids of positions t0 .. t1-1, staged once (past the table: -1)
  int* spt = reinterpret_cast<int*>(smem + dec_stage_bytes<HD, KVQ, G, NB>());
  {
    const int32_t* pt = kv.page_table + (long long)b * kv.pages_per_seq;
    const int lp0 = t0 / kv.page_size, n = (t1 - 1) / kv.page_size - lp0 + 1;
    for (int i = tid; i < n; i += 128) spt[i] = lp0 + i < kv.pages_per_seq ? pt[lp0 + i] : -1;
    __syncthreads();
  }
  const int lp0 = t0 / kv.page_size;

  // ---- one tile of K, V (and their int8 scales) into ring slot tile % NB.
  // Rows of tokens at or past t1 (or with a bad page) are zero-filled, so
  // their (masked) scores and zero probabilities meet finite values.  Each
  // thread copies the same 16-byte column of rows jb, jb + RPP, ...; page
  // arithmetic is shifts and masks when the page size is a power of two.
  constexpr int RPP = 128 / CPR, PASSES = TT / RPP;
  static_assert(128 % CPR == 0 && TT % RPP == 0, "row split of the tile copy");
  const int part = tid % CPR, jb = tid / CPR;
  const int P = kv.page_size;
  const bool pow2 = (P & (P - 1)) == 0;
  const int lgP = __ffs(P) - 1;
  auto page_of = [&](int t) { return pow2 ? t >> lgP : t / P; };
  auto slot_in_page = [&](int t) { return pow2 ? t & (P - 1) : t % P; };
  auto issue = [&](int tile) {
    const int tt0 = t0 + tile * TT;
    uint8_t* dK = sK + (tile % NB) * TT * RAWB + part * 16;
    uint8_t* dV = sV + (tile % NB) * TT * RAWB + part * 16;
#pragma unroll
    for (int k = 0; k < PASSES; ++k) {
      const int j = jb + k * RPP, t = tt0 + j;
      const int page = t < t1 ? spt[page_of(t) - lp0] : -1;
      if (page < 0 || page >= kv.n_pages) {
        if (err && t < t1) atomicExch(err, 1);
        *reinterpret_cast<uint4*>(dK + j * RAWB) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(dV + j * RAWB) = make_uint4(0, 0, 0, 0);
        continue;
      }
      const long long off = (((long long)page * Hkv + kvh) * P + slot_in_page(t)) * (I8 ? HD : HD * 2) + part * 16;
      dec_cp_async16(dK + j * RAWB, (const uint8_t*)kv.k_pool + off);
      dec_cp_async16(dV + j * RAWB, (const uint8_t*)kv.v_pool + off);
    }
    if constexpr (I8) {
      if (tid < TT) {
        const int j = tid, t = tt0 + j;
        const int page = t < t1 ? spt[page_of(t) - lp0] : -1;
        float* ks = sKs + (tile % NB) * TT + j;
        float* vs = sVs + (tile % NB) * TT + j;
        if (page < 0 || page >= kv.n_pages) {
          *ks = 0.f;
          *vs = 0.f;
        } else {
          const long long rowi = ((long long)page * Hkv + kvh) * P + slot_in_page(t);
          dec_cp_async4(ks, kv.k_scale + rowi);
          dec_cp_async4(vs, kv.v_scale + rowi);
        }
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
#pragma unroll
  for (int i = 0; i < NB - 1; ++i) {
    if (i < ntile) issue(i);
    else asm volatile("cp.async.commit_group;" ::: "memory");
  }

  // q of the G heads as the A operand: row g8 = head kvh G + g8 (rows >= G and
  // g8 + 8 are zero); bf16 as stored, or widened to fp16 for the int8 cache
  const int g8 = lane >> 2, t4 = lane & 3;
  uint32_t qa[HD / 16][4];
  {
    const uint16_t* qh = q + (long long)b * q_stride + (long long)(kvh * G + g8) * HD;
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      uint32_t lo = 0, hi = 0;
      if (g8 < G) {
        const uint16_t* qp = qh + ks * 16 + 2 * t4;  // q_stride may be odd: 16-bit loads
        lo = (uint32_t)qp[0] | ((uint32_t)qp[1] << 16);
        hi = (uint32_t)qp[8] | ((uint32_t)qp[9] << 16);
        if constexpr (I8) {
          const float2 a = bf2x2f(lo), c = bf2x2f(hi);
          lo = dec_pack<true>(a.x, a.y);
          hi = dec_pack<true>(c.x, c.y);
        }
      }
      qa[ks][0] = lo;
      qa[ks][1] = 0u;
      qa[ks][2] = hi;
      qa[ks][3] = 0u;
    }
  }
  const float scale = kLog2e * rsqrtf((float)HD);
  float o[NT][4];
#pragma unroll
  for (int i = 0; i < NT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m = -INFINITY, l = 0.f;  // row g8 (this lane's partial l)
  const int j0 = warp * 16;

  for (int tile = 0; tile < ntile; ++tile) {
    asm volatile("cp.async.wait_group %0;" ::"n"(NB - 2) : "memory");
    __syncthreads();  // tile landed for every thread; the slot refilled below is free
    if (tile + NB - 1 < ntile) issue(tile + NB - 1);
    else asm volatile("cp.async.commit_group;" ::: "memory");
    const int slot = tile % NB;
    const uint16_t* tK;
    const uint16_t* tV;
    if constexpr (I8) {
      // widen the tile's codes to fp16 (exact); scales stay per token
      const uint8_t* rk = sK + slot * TT * RAWB;
      const uint8_t* rv = sV + slot * TT * RAWB;
      for (int c = tid; c < TT * HD / 4; c += 128) {
        const int row = c / (HD / 4), col = (c % (HD / 4)) * 4;
        *reinterpret_cast<uint2*>(cK + row * LD + col) = dec_i8_to_f16x4(*reinterpret_cast<const uint32_t*>(rk + row * RAWB + col));
        *reinterpret_cast<uint2*>(cV + row * LD + col) = dec_i8_to_f16x4(*reinterpret_cast<const uint32_t*>(rv + row * RAWB + col));
      }
      __syncthreads();
      tK = cK;
      tV = cV;
    } else {
      tK = reinterpret_cast<const uint16_t*>(sK + slot * TT * RAWB);
      tV = reinterpret_cast<const uint16_t*>(sV + slot * TT * RAWB);
    }
    const int tt0 = t0 + tile * TT;
    if (tt0 + j0 < t1) {  // this warp has valid tokens in the tile (warp-uniform)
      // ---- S = Q K^T over this warp's 16 tokens: two n8 tiles
      float s[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
      for (int ks = 0; ks < HD / 16; ++ks) {
        uint32_t r[4];  // (tokens 0-7 | 8-15) x (dims lo | hi) of this k-step
        dec_ldsm_x4(r, tK + (j0 + ((lane >> 4) << 3) + (lane & 7)) * LD + ks * 16 + ((lane >> 3) & 1) * 8, false);
        dec_mma<I8>(s[0], qa[ks], r[0], r[1]);
        dec_mma<I8>(s[1], qa[ks], r[2], r[3]);
      }
      // ---- online softmax on row g8 (columns 2 t4, 2 t4 + 1 of each n8 tile)
      float sc[4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const int tok = j0 + nt * 8 + 2 * t4 + c;
          float v = s[nt][c] * scale;
          if constexpr (I8) v *= sKs[slot * TT + tok];
          sc[nt * 2 + c] = tt0 + tok < t1 ? v : -INFINITY;
        }
      float mx = fmaxf(fmaxf(sc[0], sc[1]), fmaxf(sc[2], sc[3]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float mnew = fmaxf(m, mx);
      const float ref = mnew == -INFINITY ? 0.f : mnew;
      const float corr = exp2f(m - ref);
      float p[4], ps = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        p[i] = exp2f(sc[i] - ref);
        ps += p[i];
      }
      l = l * corr + ps;
      m = mnew;
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        o[i][0] *= corr;
        o[i][1] *= corr;
      }
      if constexpr (I8) {
#pragma unroll
        for (int i = 0; i < 4; ++i) p[i] *= sVs[slot * TT + j0 + (i >> 1) * 8 + 2 * t4 + (i & 1)];
      }
      // P as the A operand over k = this warp's 16 tokens (row g8 only)
      const uint32_t pa[4] = {dec_pack<I8>(p[0], p[1]), 0u, dec_pack<I8>(p[2], p[3]), 0u};
      // ---- O += P V: V^T fragments by transposing ldmatrix, two n8 tiles per step
#pragma unroll
      for (int dn = 0; dn < HD / 16; ++dn) {
        uint32_t r[4];  // (tokens 0-7 | 8-15) x (dims +0..7 | +8..15)
        dec_ldsm_x4(r, tV + (j0 + ((lane >> 3) & 1) * 8 + (lane & 7)) * LD + dn * 16 + (lane >> 4) * 8, true);
        dec_mma<I8>(o[2 * dn], pa, r[0], r[1]);
        dec_mma<I8>(o[2 * dn + 1], pa, r[2], r[3]);
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  l += __shfl_xor_sync(0xffffffffu, l, 1);
  l += __shfl_xor_sync(0xffffffffu, l, 2);
  __syncthreads();  // the ring is reused for the merge below

  // ---- merge the 4 warps: per head, o = sum_w o_w 2^(m_w - M), l = sum_w l_w 2^(m_w - M)
  float* red = reinterpret_cast<float*>(smem);  // [4][G][HD + 2]
  if (g8 < G) {
    float* r = red + (warp * G + g8) * (HD + 2);
#pragma unroll
    for (int i = 0; i < NT; ++i) {
      r[i * 8 + 2 * t4] = o[i][0];
      r[i * 8 + 2 * t4 + 1] = o[i][1];
    }
    if (t4 == 0) {
      r[HD] = m;
      r[HD + 1] = l;
    }
  }
  __syncthreads();
  for (int i = tid; i < G * HD; i += 128) {
    const int g = i / HD, e = i % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, red[(w * G + g) * (HD + 2) + HD]);
    float ov = 0.f, L = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float* r = red + (w * G + g) * (HD + 2);
      const float f = r[HD] == -INFINITY ? 0.f : exp2f(r[HD] - M);
      ov += r[e] * f;
      L += r[HD + 1] * f;
    }
    if (splits == 1) {  // the whole context: normalise here, no combine pass
      out[((long long)b * H + kvh * G + g) * HD + e] = f2bf(ov / L);
      continue;
    }
    const long long row = ((long long)b * H + kvh * G + g) * splits + split;
    float* w = ws + row * (HD + 2);
    w[e] = ov;
    if (e == 0) {
      w[HD] = M;
      w[HD + 1] = L;
    }
  }
}

// Combine the splits of one (b, h): o = sum_s o_s 2^(m_s - M) / sum_s l_s 2^(m_s - M).
template <int HD>
__global__ void attn_combine_kernel(int H, const int32_t* __restrict__ len, int len_add, int max_len, int chunk,
                                    int splits, const float* __restrict__ ws, uint16_t* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  const int bh = blockIdx.x;
  const int b = bh / H;
  const int n = (min(len[b] + len_add, max_len) + chunk - 1) / chunk;
  const float* base = ws + (long long)bh * splits * (HD + 2);
  float M = -INFINITY;
  for (int s = 0; s < n; ++s) M = fmaxf(M, base[s * (HD + 2) + HD]);
  float L = 0.f, o = 0.f;
  const int e = threadIdx.x;
  for (int s = 0; s < n; ++s) {
    const float* w = base + s * (HD + 2);
    const float f = exp2f(w[HD] - M);
    L += w[HD + 1] * f;
    o += w[e] * f;
  }
  out[(long long)bh * HD + e] = f2bf(o / L);
}

// =====================================================================
// Decode attention over an int8 cache, head_dim 128, 16-token pages: each
// warp streams whole pages of its KV head on its own.
//
// CTA = one (sequence, KV head, context split), 4 warps; warp w takes pages
// w, w + 4, ... of the split.  A page of one KV head is 2 KB of K codes, 2 KB
// of V codes and 2 x 64 B of scales, contiguous in the pool; each warp copies
// its pages into a private 3-page cp.async ring (16-byte chunks, row r's
// chunk c stored at c ^ (r & 7) so the reads below are conflict-free) and
// waits only for its own copies: no CTA barrier inside the loop.
//
// Per page, two MMA passes (mma.sync m16n8k16, fp16 in, fp32 accumulate):
//   S^T = K Q^T: A = the page's 16 keys x 16 dims, B = Q^T (16 dims x the
//     G <= 8 query heads of the KV head): the heads fill the N = 8 of the
//     instruction.  The dims are permuted so that thread (g, t) reads 32
//     consecutive code bytes of keys g and g + 8 -- k-step ks, slots
//     (2t, 2t+1, 2t+8, 2t+9) <-> dims 32t + 4ks + (0, 1, 2, 3) -- and Q is
//     loaded with the same permutation once per CTA.
//   O^T += V^T P'^T: A = 16 dims x the page's 16 tokens (thread (g, t) owns
//     dims 16g .. 16g + 15, so it reads one 16-byte chunk of each of its four
//     tokens; m-tile mt holds dims 16g + 2mt and 16g + 2mt + 1), B = P' (the
//     probabilities times each token's V scale) of 16 tokens x 8 heads, moved
//     from the S^T accumulator layout by four shuffles.
// Codes enter as fp16(1152 + q) (a byte permute with 0x64 high bytes after
// q ^ 0x80, exact); the offset is removed in fp32: scores subtract
// 1152 sum_d Q[h][d], outputs 1152 sum_t P'[t][h].  Online softmax in the
// log2 domain per head, the K scales multiplying the score columns.  The
// warps are merged in shared memory at the end; the result is normalised in
// place (one split) or written as (o, m, l) for attn_combine_kernel.
// =====================================================================
constexpr int kD8Warps = 4, kD8Stages = 3;
constexpr int kD8PageBytes = 2 * 16 * 128 + 2 * 16 * 4;  // K and V codes, then K and V scales

FP_DEV uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t r;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
  return r;
}
FP_DEV uint4 lds128(const uint8_t* p) { return *reinterpret_cast<const uint4*>(p); }
FP_DEV uint32_t word4(const uint4& v, int i) { return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w; }

constexpr size_t d8_smem_bytes(int chunk) {
  return (size_t)kD8Warps * kD8Stages * kD8PageBytes + ((size_t)chunk / 16 + 2) * sizeof(int);
}

template <int G>
__global__ void __launch_bounds__(kD8Warps * 32) attn_decode_i8_kernel(
    const uint16_t* __restrict__ q, int q_stride, int H, fp_kv_view kv, const int32_t* __restrict__ len,
    int len_add, int max_len, int chunk, int splits, float* __restrict__ ws, uint16_t* __restrict__ out,
    int32_t* err) {
  constexpr int HD = 128;
  extern __shared__ __align__(16) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  // no early trigger: the linear after it takes whole SMs, and launched early
  // its CTAs would sit beside these and stream weights while they stream the cache
  pdl_wait();
  const int Hkv = kv.n_kv_heads;
  const int b = blockIdx.x / Hkv, kvh = blockIdx.x % Hkv;
  const int split = blockIdx.y;
  int T = len[b] + len_add;
  if (T > max_len) {  // never past the positions the grid and the page table cover
    if (err && split == 0 && threadIdx.x == 0) atomicExch(err, 1);
    T = max_len;
  }
  const int t0 = split * chunk;
  if (t0 >= T) {
    if (splits == 1)  // empty context: zero output
      for (int i = threadIdx.x; i < G * HD; i += blockDim.x) out[((long long)b * H + kvh * G) * HD + i] = 0;
    return;
  }
  const int t1 = min(T, t0 + chunk);
  const int np = (t1 - t0 + 15) / 16;  // pages of the split (t0 is a multiple of 64)
  // ---- the split's page ids, staged once (past the table: -1)
  int* spt = reinterpret_cast<int*>(smem + kD8Warps * kD8Stages * kD8PageBytes);
  {
    const int32_t* pt = kv.page_table + (long long)b * kv.pages_per_seq;
    const int lp0 = t0 / 16;
    for (int i = threadIdx.x; i < np; i += blockDim.x) spt[i] = lp0 + i < kv.pages_per_seq ? pt[lp0 + i] : -1;
    __syncthreads();
  }
  uint8_t* ring = smem + warp * kD8Stages * kD8PageBytes;

  // ---- copy page j of this warp (split page warp + 4 j) into ring slot j % 3
  auto issue = [&](int j) {
    const int pi = warp + kD8Warps * j;
    uint8_t* dst = ring + (j % kD8Stages) * kD8PageBytes;
    if (pi < np) {
      const int page = spt[pi];
      if (page >= 0 && page < kv.n_pages) {
        const long long row0 = ((long long)page * Hkv + kvh) * 16;  // first token row of (page, head)
        const uint8_t* kg = (const uint8_t*)kv.k_pool + row0 * HD;
        const uint8_t* vg = (const uint8_t*)kv.v_pool + row0 * HD;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int c = lane + 32 * i, r = c >> 3, cc = c & 7;
          const int off = r * HD + ((cc ^ (r & 7)) << 4);
          dec_cp_async16(dst + off, kg + c * 16);
          dec_cp_async16(dst + 2048 + off, vg + c * 16);
        }
        if (lane < 4) dec_cp_async16(dst + 4096 + lane * 16, (const uint8_t*)(kv.k_scale + row0) + lane * 16);
        else if (lane < 8) dec_cp_async16(dst + 4160 + (lane - 4) * 16, (const uint8_t*)(kv.v_scale + row0) + (lane - 4) * 16);
      } else {
        // a bad page id reads as zero codes and zero scales
        if (err && lane == 0) atomicExch(err, 1);
        for (int i = lane; i < kD8PageBytes / 16; i += 32) *reinterpret_cast<uint4*>(dst + i * 16) = make_uint4(0, 0, 0, 0);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  const int nj = np > warp ? (np - warp + kD8Warps - 1) / kD8Warps : 0;  // this warp's pages
#pragma unroll
  for (int j = 0; j < kD8Stages - 1; ++j) issue(j);

  // ---- Q^T as the B operand (head g, dims 32t + 4ks + 0..3), fp16; and
  // sum_d Q[h][d] of the fp16 values for the heads 2t, 2t + 1 of this thread
  uint32_t qb[8][2];
  float qsum = 0.f;
  {
    const uint16_t* qh = q + (long long)b * q_stride + (long long)(kvh * G + g) * HD + 32 * t;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      uint32_t lo = 0, hi = 0;
      if (g < G) {  // q_stride may be odd: 16-bit loads
        const uint16_t* qp = qh + 4 * ks;
        const __half2 a = __floats2half2_rn(bf2f(qp[0]), bf2f(qp[1]));
        const __half2 c = __floats2half2_rn(bf2f(qp[2]), bf2f(qp[3]));
        const float2 fa = __half22float2(a), fc = __half22float2(c);
        qsum += (fa.x + fa.y) + (fc.x + fc.y);
        lo = *reinterpret_cast<const uint32_t*>(&a);
        hi = *reinterpret_cast<const uint32_t*>(&c);
      }
      qb[ks][0] = lo;
      qb[ks][1] = hi;
    }
    qsum += __shfl_xor_sync(0xffffffffu, qsum, 1);
    qsum += __shfl_xor_sync(0xffffffffu, qsum, 2);
  }
  // lanes 4h .. 4h + 3 hold head h's sum; this thread's score columns are heads 2t, 2t + 1
  const float qoff0 = 1152.f * __shfl_sync(0xffffffffu, qsum, 8 * t);
  const float qoff1 = 1152.f * __shfl_sync(0xffffffffu, qsum, 8 * t + 4);
  const float scale = kLog2e * rsqrtf((float)HD);

  float o[8][4];  // O^T: m-tile mt rows (dims 16g + 2mt, 16g + 2mt + 1) x heads (2t, 2t + 1)
#pragma unroll
  for (int i = 0; i < 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f}, sp[2] = {0.f, 0.f};  // heads 2t, 2t + 1
  const uint32_t sw = (uint32_t)(g & 7);

  for (int j = 0; j < nj; ++j) {
    asm volatile("cp.async.wait_group %0;" ::"n"(kD8Stages - 2) : "memory");
    __syncwarp();  // every lane's copies of page j landed; the slot refilled below was read last round
    issue(j + kD8Stages - 1);
    const uint8_t* pg = ring + (j % kD8Stages) * kD8PageBytes;
    const int tok0 = t0 + (warp + kD8Warps * j) * 16;

    // ---- S^T = K Q^T over the page's 16 tokens
    float s[4] = {0.f, 0.f, 0.f, 0.f};  // (token g | g + 8) x (head 2t | 2t + 1)
    {
      const uint4 ka0 = lds128(pg + g * HD + (((2 * t) ^ sw) << 4));
      const uint4 ka1 = lds128(pg + g * HD + (((2 * t + 1) ^ sw) << 4));
      const uint4 kb0 = lds128(pg + (g + 8) * HD + (((2 * t) ^ sw) << 4));
      const uint4 kb1 = lds128(pg + (g + 8) * HD + (((2 * t + 1) ^ sw) << 4));
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const uint32_t wa = word4(ks < 4 ? ka0 : ka1, ks & 3) ^ 0x80808080u;
        const uint32_t wb = word4(ks < 4 ? kb0 : kb1, ks & 3) ^ 0x80808080u;
        const uint32_t a[4] = {prmt(wa, 0x64646464u, 0x5140), prmt(wb, 0x64646464u, 0x5140),
                               prmt(wa, 0x64646464u, 0x5342), prmt(wb, 0x64646464u, 0x5342)};
        dec_mma<true>(s, a, qb[ks][0], qb[ks][1]);
      }
    }
    // ---- scores (log2 domain): s_k[token] (S^T - 1152 sum Q) / sqrt(hd); tokens past t1 masked
    const float* ksc = reinterpret_cast<const float*>(pg + 4096);
    const float* vsc = reinterpret_cast<const float*>(pg + 4160);
    const bool ok_lo = tok0 + g < t1, ok_hi = tok0 + g + 8 < t1;
    const float sk_lo = ksc[g] * scale, sk_hi = ksc[g + 8] * scale;
    float sc[4];
    sc[0] = ok_lo ? (s[0] - qoff0) * sk_lo : -INFINITY;
    sc[1] = ok_lo ? (s[1] - qoff1) * sk_lo : -INFINITY;
    sc[2] = ok_hi ? (s[2] - qoff0) * sk_hi : -INFINITY;
    sc[3] = ok_hi ? (s[3] - qoff1) * sk_hi : -INFINITY;
    uint32_t pk[2];  // fp16 pairs (P'[token g][head 2t + e], P'[token g + 8][head 2t + e])
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      float mx = fmaxf(sc[e], sc[2 + e]);
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
      const float mnew = fmaxf(m[e], mx);
      const float ref = mnew == -INFINITY ? 0.f : mnew;
      const float corr = exp2f(m[e] - ref);
      const float p_lo = exp2f(sc[e] - ref), p_hi = exp2f(sc[2 + e] - ref);
      l[e] = l[e] * corr + p_lo + p_hi;
      m[e] = mnew;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        o[mt][e] *= corr;
        o[mt][2 + e] *= corr;
      }
      // P' = P times the token's V scale (zero for masked tokens), rounded to fp16;
      // the V offset uses the sum of the rounded values
      const __half2 pp = __floats2half2_rn(ok_lo ? p_lo * vsc[g] : 0.f, ok_hi ? p_hi * vsc[g + 8] : 0.f);
      const float2 pr = __half22float2(pp);
      sp[e] = sp[e] * corr + pr.x + pr.y;
      pk[e] = *reinterpret_cast<const uint32_t*>(&pp);
    }
    // ---- P'^T as the B operand: thread (g, t) needs head g at tokens 2t, 2t + 1
    // (from lane 8t + g/2) and 2t + 8, 2t + 9 (lane 8t + 4 + g/2), parity g & 1
    uint32_t pb0, pb1;
    {
      const int l0 = 8 * t + (g >> 1), l1 = l0 + 4;
      const uint32_t a0 = __shfl_sync(0xffffffffu, pk[0], l0), a1 = __shfl_sync(0xffffffffu, pk[1], l0);
      const uint32_t c0 = __shfl_sync(0xffffffffu, pk[0], l1), c1 = __shfl_sync(0xffffffffu, pk[1], l1);
      const uint32_t v0 = (g & 1) ? a1 : a0, v1 = (g & 1) ? c1 : c0;  // (tok 2t | 2t+8), (tok 2t+1 | 2t+9)
      pb0 = prmt(v0, v1, 0x5410);  // tokens 2t, 2t + 1
      pb1 = prmt(v0, v1, 0x7632);  // tokens 2t + 8, 2t + 9
    }
    // ---- O^T += V^T P'^T: thread (g, t) reads dims 16g .. 16g + 15 of tokens 2t, 2t + 1, 2t + 8, 2t + 9
    {
      const uint4 va = lds128(pg + 2048 + (2 * t) * HD + ((g ^ ((2 * t) & 7)) << 4));
      const uint4 vb = lds128(pg + 2048 + (2 * t + 1) * HD + ((g ^ ((2 * t + 1) & 7)) << 4));
      const uint4 vc = lds128(pg + 2048 + (2 * t + 8) * HD + ((g ^ ((2 * t + 8) & 7)) << 4));
      const uint4 vd = lds128(pg + 2048 + (2 * t + 9) * HD + ((g ^ ((2 * t + 9) & 7)) << 4));
#pragma unroll
      for (int wi = 0; wi < 4; ++wi) {
        const uint32_t A = word4(va, wi) ^ 0x80808080u, Bw = word4(vb, wi) ^ 0x80808080u;
        const uint32_t C = word4(vc, wi) ^ 0x80808080u, D = word4(vd, wi) ^ 0x80808080u;
#pragma unroll
        for (int h = 0; h < 2; ++h) {  // m-tile 2 wi + h: bytes 2h, 2h + 1 of the words
          const uint32_t xab = prmt(A, Bw, h ? 0x7362 : 0x5140), xcd = prmt(C, D, h ? 0x7362 : 0x5140);
          const uint32_t a[4] = {prmt(xab, 0x64646464u, 0x5140), prmt(xab, 0x64646464u, 0x5342),
                                 prmt(xcd, 0x64646464u, 0x5140), prmt(xcd, 0x64646464u, 0x5342)};
          dec_mma<true>(o[2 * wi + h], a, pb0, pb1);
        }
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
#pragma unroll
  for (int e = 0; e < 2; ++e) {
#pragma unroll
    for (int x = 4; x <= 16; x <<= 1) {
      l[e] += __shfl_xor_sync(0xffffffffu, l[e], x);
      sp[e] += __shfl_xor_sync(0xffffffffu, sp[e], x);
    }
  }
  __syncthreads();  // the rings are reused for the merge below

  // ---- merge the 4 warps: per head, o = sum_w o_w 2^(m_w - M), l = sum_w l_w 2^(m_w - M)
  float* red = reinterpret_cast<float*>(smem);  // [4][8][HD + 2]
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int hh = 2 * t + e;
    if (hh < G) {
      float* r = red + (warp * 8 + hh) * (HD + 2);
      const float off = 1152.f * sp[e];
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        r[16 * g + 2 * mt] = o[mt][e] - off;
        r[16 * g + 2 * mt + 1] = o[mt][2 + e] - off;
      }
      if (g == 0) {
        r[HD] = m[e];
        r[HD + 1] = l[e];
      }
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < G * HD; i += blockDim.x) {
    const int hh = i / HD, e = i % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kD8Warps; ++w) M = fmaxf(M, red[(w * 8 + hh) * (HD + 2) + HD]);
    float ov = 0.f, L = 0.f;
#pragma unroll
    for (int w = 0; w < kD8Warps; ++w) {
      const float* r = red + (w * 8 + hh) * (HD + 2);
      const float f = r[HD] == -INFINITY ? 0.f : exp2f(r[HD] - M);
      ov += r[e] * f;
      L += r[HD + 1] * f;
    }
    if (splits == 1) {  // the whole context: normalise here, no combine pass
      out[((long long)b * H + kvh * G + hh) * HD + e] = f2bf(ov / L);
      continue;
    }
    const long long row = ((long long)b * H + kvh * G + hh) * splits + split;
    float* w = ws + row * (HD + 2);
    w[e] = ov;
    if (e == 0) {
      w[HD] = M;
      w[HD + 1] = L;
    }
  }
}

template <int G>
static cudaError_t launch_decode_i8(const uint16_t* q, int q_stride, int B, int H, const fp_kv_view& kv,
                                    const int32_t* len, int len_add, int max_len, DecodeGeom g, float* ws,
                                    uint16_t* out, int32_t* err, cudaStream_t s, cudaError_t* second) {
  const size_t smem = d8_smem_bytes(g.chunk);
  auto kern = attn_decode_i8_kernel<G>;
  static std::atomic<unsigned long long> attr{0};
  FP_CUDA_TRY(smem_limit_once(kern, (int)d8_smem_bytes(kDecMaxChunkTiles * kDecTT), &attr));
  dim3 grid(B * kv.n_kv_heads, g.splits);
  cudaError_t e = launch(kern, grid, dim3(kD8Warps * 32), smem, s, q, q_stride, H, kv, len, len_add, max_len,
                         g.chunk, g.splits, ws, out, err);
  if (e != cudaSuccess || g.splits == 1) return e;
  e = launch(attn_combine_kernel<128>, dim3(B * H), dim3(128), 0, s, H, len, len_add, max_len, g.chunk, g.splits,
             (const float*)ws, out);
  if (second) *second = e;
  return e;
}

template <int HD, int KVQ, int G, int NB>
static cudaError_t launch_decode_nb(const uint16_t* q, int q_stride, int B, int H, const fp_kv_view& kv,
                                    const int32_t* len, int len_add, int max_len, DecodeGeom g, float* ws,
                                    uint16_t* out, int32_t* err, cudaStream_t s, cudaError_t* second) {
  // the ring also holds the 4-warp merge buffer after the loop
  const size_t smem = dec_stage_bytes<HD, KVQ, G, NB>() + ((size_t)g.chunk / kv.page_size + 2) * sizeof(int);
  auto kern = attn_decode_kernel<HD, KVQ, G, NB>;
  if (smem > 48 * 1024) FP_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  dim3 grid(B * kv.n_kv_heads, g.splits);
  cudaError_t e = launch(kern, grid, dim3(128), smem, s, q, q_stride, H, kv, len, len_add, max_len, g.chunk,
                         g.splits, ws, out, err);
  if (e != cudaSuccess || g.splits == 1) return e;
  e = launch(attn_combine_kernel<HD>, dim3(B * H), dim3(HD), 0, s, H, len, len_add, max_len, g.chunk, g.splits,
             (const float*)ws, out);
  if (second) *second = e;
  return e;
}

template <int HD, int KVQ, int G>
static cudaError_t launch_decode_t(const uint16_t* q, int q_stride, int B, int H, const fp_kv_view& kv,
                                   const int32_t* len, int len_add, int max_len, DecodeGeom g, float* ws,
                                   uint16_t* out, int32_t* err, cudaStream_t s, cudaError_t* second) {
  return g.nb == 2 ? launch_decode_nb<HD, KVQ, G, 2>(q, q_stride, B, H, kv, len, len_add, max_len, g, ws, out, err, s, second)
                   : launch_decode_nb<HD, KVQ, G, 3>(q, q_stride, B, H, kv, len, len_add, max_len, g, ws, out, err, s, second);
}

template <int HD, int KVQ>
static cudaError_t launch_decode_g(int G, const uint16_t* q, int q_stride, int B, int H, const fp_kv_view& kv,
                                   const int32_t* len, int len_add, int max_len, DecodeGeom g, float* ws,
                                   uint16_t* out, int32_t* err, cudaStream_t s, cudaError_t* second) {
  switch (G) {
    case 1: return launch_decode_t<HD, KVQ, 1>(q, q_stride, B, H, kv, len, len_add, max_len, g, ws, out, err, s, second);
    case 2: return launch_decode_t<HD, KVQ, 2>(q, q_stride, B, H, kv, len, len_add, max_len, g, ws, out, err, s, second);
    case 4: return launch_decode_t<HD, KVQ, 4>(q, q_stride, B, H, kv, len, len_add, max_len, g, ws, out, err, s, second);
    case 8: return launch_decode_t<HD, KVQ, 8>(q, q_stride, B, H, kv, len, len_add, max_len, g, ws, out, err, s, second);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_attention_decode(const uint16_t* q, int q_stride, int B, int n_heads, const fp_kv_view& kv,
                                    const int32_t* len, int len_add, int max_len, uint16_t* out, void* ws,
                                    int32_t* err, cudaStream_t s, cudaError_t* second) {
  const int G = n_heads / kv.n_kv_heads;
  float* w = (float*)ws;
  const bool a16 = (((uintptr_t)kv.k_pool | (uintptr_t)kv.v_pool | (uintptr_t)kv.k_scale | (uintptr_t)kv.v_scale) & 15) == 0;
  if (dec_i8_shape(kv.kvquant, kv.head_dim, kv.page_size) && a16) {
    const DecodeGeom g = decode_geom_for(B, kv.n_kv_heads, kv.head_dim, kv.kvquant, kv.page_size, max_len);
    switch (G) {
      case 1: return launch_decode_i8<1>(q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second);
      case 2: return launch_decode_i8<2>(q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second);
      case 4: return launch_decode_i8<4>(q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second);
      case 8: return launch_decode_i8<8>(q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second);
      default: return cudaErrorInvalidValue;
    }
  }
  const DecodeGeom g = decode_geom(B, kv.n_kv_heads, max_len);
  if (kv.head_dim == 64) {
    return kv.kvquant == FP_KV_BF16
               ? launch_decode_g<64, FP_KV_BF16>(G, q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second)
               : launch_decode_g<64, FP_KV_INT8>(G, q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second);
  }
  return kv.kvquant == FP_KV_BF16
             ? launch_decode_g<128, FP_KV_BF16>(G, q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second)
             : launch_decode_g<128, FP_KV_INT8>(G, q, q_stride, B, n_heads, kv, len, len_add, max_len, g, w, out, err, s, second);
}

// =====================================================================
// Prefill: causal attention of S query rows per sequence against cache
// positions 0..S-1.  CTA = 64 query rows of one (b, h); 4 warps x 16 rows;
// key/value tiles of 64 stream through a two-stage cp.async ring (the next
// tile loads while this one computes) for bf16 caches; int8 codes are loaded
// and widened exactly to bf16 tile by tile (a staged copy of the codes plus
// a widening pass measured slower at the 70B shape), their per-token scales
// multiplying S and P.  S = Q K^T and O += P V with mma.sync m16n8k16 (bf16
// in, fp32 accumulate; ldmatrix, transposed for V) and an online
// softmax in the log2 domain; P stays in registers as the A operand.
// =====================================================================
FP_DEV void mma_bf16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

FP_DEV void ldsm_x4(uint32_t* r, const void* p) {
  uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}

FP_DEV void ldsm_x2(uint32_t& r0, uint32_t& r1, const void* p) {
  uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(a));
}

FP_DEV void ldsm_x2_trans(uint32_t& r0, uint32_t& r1, const void* p) {
  uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(a));
}

// 16-byte cp.async that writes zeros when `valid` is false (source size 0).
FP_DEV void pf_cp16(void* smem, const void* gmem, bool valid) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(s), "l"(gmem), "r"(valid ? 16 : 0) : "memory");
}

template <int HD, int KVQ>
constexpr size_t prefill_smem_bytes() {
  constexpr int BT = 64, LD = HD + 8;
  // bf16 cache: two stages of K and V tiles; int8 cache: one K and V tile
  // and the tile's scales.  The Q tile borrows a K tile.
  if (KVQ == FP_KV_INT8) return (size_t)2 * BT * LD * 2 + (size_t)2 * BT * sizeof(float);
  return (size_t)2 * 2 * BT * LD * 2;
}

template <int HD, int KVQ>
__global__ void __launch_bounds__(128) attn_prefill_kernel(const uint16_t* __restrict__ q, int q_stride, int S,
                                                           int H, fp_kv_view kv, uint16_t* __restrict__ out,
                                                           int32_t* err) {
  constexpr int BT = 64;        // query rows per CTA and keys per tile
  constexpr int LD = HD + 8;    // padded row (bf16 elements) against ldmatrix bank conflicts
  constexpr bool I8 = KVQ == FP_KV_INT8;
  constexpr int RB = I8 ? HD : 2 * HD;  // bytes of one cached row
  constexpr int CPR = RB / 16;          // 16-byte chunks per cached row
  extern __shared__ __align__(16) uint8_t smem_raw[];
  pdl_trigger();
  pdl_wait();
  constexpr int NT = I8 ? 1 : 2;  // bf16 tile stages
  uint16_t* sKV = reinterpret_cast<uint16_t*>(smem_raw);  // [stage][K | V][BT][LD] bf16
  float* rsc = reinterpret_cast<float*>(sKV + NT * 2 * BT * LD);  // int8: [K | V][BT] scales
  auto tileK = [&](int st) { return sKV + ((st % NT) * 2 + 0) * BT * LD; };
  auto tileV = [&](int st) { return sKV + ((st % NT) * 2 + 1) * BT * LD; };
  // the Q tile is read into fragments before the first __syncthreads of the
  // key loop, after which that K tile is first written
  uint16_t* sQ = tileK(1);

  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int Hkv = kv.n_kv_heads, G = H / Hkv, kvh = h / G;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g8 = lane >> 2, t4 = lane & 3;
  const int q0 = qt * BT;
  const int32_t* pt = kv.page_table + (long long)b * kv.pages_per_seq;
  const int last_key = min(q0 + BT, S) - 1;
  const int ntile = last_key / BT + 1;

  // ---- cache row of key t: its index in the pool, or -1 past S / on a bad page
  auto row_of = [&](int t) -> long long {
    if (t >= S) return -1;
    const int page = pt[t / kv.page_size];
    if (page < 0 || page >= kv.n_pages) {
      if (err) atomicExch(err, 1);
      return -1;
    }
    return ((long long)page * Hkv + kvh) * kv.page_size + t % kv.page_size;
  };
  // ---- bf16: one key tile (rows k0 .. k0 + 63, zeros where row_of < 0) into stage st
  auto issue = [&](int tile, int st) {
    if constexpr (!I8) {
      const int k0 = tile * BT;
      for (int c = tid; c < 2 * BT * CPR; c += 128) {
        const int which = c / (BT * CPR), r = (c % (BT * CPR)) / CPR, cc = c % CPR;
        const long long rowi = row_of(k0 + r);
        const uint8_t* src = (const uint8_t*)(which ? kv.v_pool : kv.k_pool) + (rowi >= 0 ? rowi * RB + cc * 16 : 0);
        pf_cp16((which ? tileV(st) : tileK(st)) + r * LD + cc * 8, src, rowi >= 0);
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
  };
  issue(0, 0);

  // ---- Q tile -> fragments (row-major A operand of the warp's 16 rows)
  constexpr int QCPR = HD / 8;
  for (int c = tid; c < BT * QCPR; c += 128) {
    const int r = c / QCPR, cc = c % QCPR;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (q0 + r < S) v = ld_nc16(q + ((long long)b * S + q0 + r) * q_stride + (long long)h * HD + cc * 8);
    *reinterpret_cast<uint4*>(sQ + r * LD + cc * 8) = v;
  }
  __syncthreads();
  uint32_t qf[HD / 16][4];
  {
    const int r = warp * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
    const int c = 8 * (lane >> 4);
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) ldsm_x4(qf[kk], sQ + r * LD + kk * 16 + c);
  }

  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  const float scale = kLog2e * rsqrtf((float)HD);
  const int qrow0 = q0 + warp * 16 + g8;  // rows qrow0 and qrow0 + 8

  for (int tile = 0; tile < ntile; ++tile) {
    const int st = tile & 1, k0 = tile * BT;
    if constexpr (!I8) asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();  // the tile landed for every thread; every warp is done with the other stage
    if (tile + 1 < ntile) issue(tile + 1, st ^ 1);
    const float* sks = rsc;
    const float* svs = rsc + BT;
    if constexpr (I8) {
      // codes -> bf16 (small integers: exact) while loading; the scales multiply S and P
      for (int c = tid; c < 2 * BT * CPR; c += 128) {
        const int which = c / (BT * CPR), r = (c % (BT * CPR)) / CPR, cc = c % CPR;
        const long long rowi = row_of(k0 + r);
        uint4 v = make_uint4(0, 0, 0, 0);
        float sc = 0.f;
        if (rowi >= 0) {
          v = ld_nc16((const uint8_t*)(which ? kv.v_pool : kv.k_pool) + rowi * RB + cc * 16);
          sc = (which ? kv.v_scale : kv.k_scale)[rowi];
        }
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
        uint32_t o8[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const uint32_t word = w[i >> 1];
          const int sh = 16 * (i & 1);
          o8[i] = pack_bf2((float)(int8_t)((word >> sh) & 0xFF), (float)(int8_t)((word >> (sh + 8)) & 0xFF));
        }
        uint16_t* dst = (which ? tileV(st) : tileK(st)) + r * LD + cc * 16;
        *reinterpret_cast<uint4*>(dst) = make_uint4(o8[0], o8[1], o8[2], o8[3]);
        *reinterpret_cast<uint4*>(dst + 8) = make_uint4(o8[4], o8[5], o8[6], o8[7]);
        if (cc == 0) rsc[which * BT + r] = sc;
      }
      __syncthreads();
    }
    const uint16_t* tK = tileK(st);
    const uint16_t* tV = tileV(st);
    // ---- S = Q K^T for this warp's 16 rows x 64 keys (two-matrix ldmatrix per
    // n8 key tile: the four-matrix form measured 25% slower with the int8 cache)
    float sacc[BT / 8][4];
#pragma unroll
    for (int n = 0; n < BT / 8; ++n) sacc[n][0] = sacc[n][1] = sacc[n][2] = sacc[n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int n = 0; n < BT / 8; ++n) {
        uint32_t b0, b1;
        ldsm_x2(b0, b1, tK + (n * 8 + (lane & 7)) * LD + kk * 16 + 8 * ((lane >> 3) & 1));
        mma_bf16(sacc[n], qf[kk], b0, b1);
      }
    }
    // ---- scale, mask, online softmax
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int n = 0; n < BT / 8; ++n) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int key = k0 + n * 8 + 2 * t4 + (i & 1);
        const int row = qrow0 + 8 * (i >> 1);
        float v = sacc[n][i] * scale;
        if constexpr (I8) v *= sks[n * 8 + 2 * t4 + (i & 1)];
        if (key > row || key >= S) v = -INFINITY;
        sacc[n][i] = v;
        mx[i >> 1] = fmaxf(mx[i >> 1], v);
      }
    }
    float corr[2], mref[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      const float mnew = fmaxf(mrow[r], mx[r]);
      mref[r] = mnew == -INFINITY ? 0.f : mnew;
      corr[r] = exp2f(mrow[r] - mref[r]);
      mrow[r] = mnew;
      lrow[r] *= corr[r];
    }
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      o[i][0] *= corr[0];
      o[i][1] *= corr[0];
      o[i][2] *= corr[1];
      o[i][3] *= corr[1];
    }
    uint32_t pa[BT / 16][4];
#pragma unroll
    for (int n = 0; n < BT / 8; ++n) {
      float p[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        p[i] = exp2f(sacc[n][i] - mref[i >> 1]);
        lrow[i >> 1] += p[i];
        if constexpr (I8) p[i] *= svs[n * 8 + 2 * t4 + (i & 1)];
      }
      pa[n >> 1][(n & 1) * 2 + 0] = pack_bf2(p[0], p[1]);
      pa[n >> 1][(n & 1) * 2 + 1] = pack_bf2(p[2], p[3]);
    }
    // ---- O += P V: V^T fragments by transposing ldmatrix
#pragma unroll
    for (int j = 0; j < BT / 16; ++j) {
#pragma unroll
      for (int dt = 0; dt < HD / 8; ++dt) {
        uint32_t b0, b1;
        ldsm_x2_trans(b0, b1, tV + (j * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * LD + dt * 8);
        mma_bf16(o[dt], pa[j], b0, b1);
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  // ---- normalise and store
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int row = qrow0 + 8 * r;
    if (row >= S) continue;
    const float inv = 1.f / lrow[r];
    uint16_t* dst = out + ((long long)b * S + row) * ((long long)H * HD) + (long long)h * HD;
#pragma unroll
    for (int dt = 0; dt < HD / 8; ++dt) {
      *reinterpret_cast<uint32_t*>(dst + dt * 8 + 2 * t4) = pack_bf2(o[dt][2 * r] * inv, o[dt][2 * r + 1] * inv);
    }
  }
}

template <int HD, int KVQ>
static cudaError_t launch_prefill_t(const uint16_t* q, int q_stride, int B, int S, int H, const fp_kv_view& kv,
                                    uint16_t* out, int32_t* err, cudaStream_t s) {
  const size_t smem = prefill_smem_bytes<HD, KVQ>();
  auto kern = attn_prefill_kernel<HD, KVQ>;
  static bool attr = false;
  if (!attr) {
    FP_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    attr = true;
  }
  dim3 grid((S + 63) / 64, H, B);
  return launch(kern, grid, dim3(128), smem, s, q, q_stride, S, H, kv, out, err);
}

cudaError_t launch_attention_prefill(const uint16_t* q, int q_stride, int B, int S, int n_heads,
                                     const fp_kv_view& kv, uint16_t* out, int32_t* err, cudaStream_t s) {
  if (B <= 0 || S <= 0) return cudaSuccess;
  if (attention_prefill_tc_ok(B, S, n_heads, kv, q, q_stride))
    return launch_attention_prefill_tc(q, q_stride, B, S, n_heads, kv, out, err, s);
  if (kv.head_dim == 64)
    return kv.kvquant == FP_KV_BF16 ? launch_prefill_t<64, FP_KV_BF16>(q, q_stride, B, S, n_heads, kv, out, err, s)
                                    : launch_prefill_t<64, FP_KV_INT8>(q, q_stride, B, S, n_heads, kv, out, err, s);
  return kv.kvquant == FP_KV_BF16 ? launch_prefill_t<128, FP_KV_BF16>(q, q_stride, B, S, n_heads, kv, out, err, s)
                                  : launch_prefill_t<128, FP_KV_INT8>(q, q_stride, B, S, n_heads, kv, out, err, s);
}

}  // namespace fpk
