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

#include "common.cuh"
#include "kernels.cuh"

namespace fpk {

static constexpr float kLog2e = 1.4426950408889634f;

// =====================================================================
// Decode: grid (B * Hkv, splits); one CTA handles the G = H / Hkv query
// heads of one KV head over one chunk of the context.  The chunk's K and V
// stream through a ring of 32-token tiles in shared memory (cp.async, two
// tiles in flight); each warp takes 8 tokens of a tile and keeps its own
// online softmax, and the 4 warps are merged at the end.
// =====================================================================
constexpr int kDecTile = 32;  // tokens per tile: two 16-token pages
constexpr int kDecBuf = 3;    // ring depth
constexpr int kDecOcc = 4;    // resident CTAs per SM assumed by the split geometry

struct DecodeGeom {
  int chunk;   // positions per split (multiple of kDecTile)
  int splits;  // ceil(max_len / chunk)
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

// As many splits as fill the resident CTA slots once (whole waves), at least
// one tile per split.  Splits never grow with n_kv_heads, so the workspace
// sized for n_kv_heads = 1 covers every launch.
static DecodeGeom decode_geom(int B, int n_kv_heads, int max_len) {
  const long long pairs = (long long)B * n_kv_heads;
  const long long slots = (long long)dec_sm_count() * kDecOcc;
  const int tiles = (max_len + kDecTile - 1) / kDecTile;
  int splits = (int)std::max<long long>(1, slots / pairs);
  splits = std::min(splits, tiles);
  const int per_tiles = (tiles + splits - 1) / splits;
  DecodeGeom g;
  g.chunk = per_tiles * kDecTile;
  g.splits = (max_len + g.chunk - 1) / g.chunk;
  return g;
}

size_t attention_decode_ws_bytes(int B, int n_heads, int head_dim, int max_len) {
  DecodeGeom g = decode_geom(B, 1, max_len);
  size_t rows = (size_t)B * n_heads * g.splits;
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

template <int HD, int KVQ>
constexpr size_t dec_smem_bytes() {
  return (size_t)kDecBuf * kDecTile * HD * (KVQ == FP_KV_BF16 ? 2 : 1) * 2 +
         (KVQ == FP_KV_INT8 ? (size_t)kDecBuf * kDecTile * 2 * sizeof(float) : 0);
}

// Workspace layout for (b, h, split): o [HD] fp32 (un-normalised, relative to
// m), then (m, l) in the log2 domain.
template <int HD, int KVQ, int G>
__global__ void __launch_bounds__(128) attn_decode_kernel(const uint16_t* __restrict__ q, int q_stride, int H,
                                                          fp_kv_view kv, const int32_t* __restrict__ len,
                                                          int len_add, int max_len, int chunk, int splits,
                                                          float* __restrict__ ws, int32_t* err) {
  constexpr int TT = kDecTile, NBUF = kDecBuf;
  constexpr int ELT = KVQ == FP_KV_BF16 ? 2 : 1, ROWB = HD * ELT, TILEB = TT * ROWB, CPR = ROWB / 16;
  constexpr int DPL = HD / 32;                   // dims per lane
  constexpr int TG = G >= 4 ? 2 : (G == 2 ? 4 : 8);  // tokens per softmax update
  extern __shared__ __align__(16) uint8_t smem[];
  uint8_t* sK = smem;                  // [NBUF][TT][ROWB]
  uint8_t* sV = sK + NBUF * TILEB;     // [NBUF][TT][ROWB]
  float* sKs = reinterpret_cast<float*>(sV + NBUF * TILEB);  // int8: [NBUF][TT]
  float* sVs = sKs + NBUF * TT;
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
  if (t0 >= T) return;
  const int t1 = min(T, t0 + chunk);
  const int ntile = (t1 - t0 + TT - 1) / TT;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int32_t* pt = kv.page_table + (long long)b * kv.pages_per_seq;

  // ---- issue one tile of K, V (and their int8 scales) into ring slot tile % NBUF
  auto issue = [&](int tile) {
    const int tt0 = t0 + tile * TT;
    uint8_t* dK = sK + (tile % NBUF) * TILEB;
    uint8_t* dV = sV + (tile % NBUF) * TILEB;
    for (int c = tid; c < TT * CPR; c += 128) {
      const int j = c / CPR, part = c % CPR, t = tt0 + j;
      const int lp = t / kv.page_size;
      if (lp >= kv.pages_per_seq) continue;  // past the sequence's table: masked below
      const int page = pt[lp];
      uint8_t* dk = dK + j * ROWB + part * 16;
      uint8_t* dv = dV + j * ROWB + part * 16;
      if (page < 0 || page >= kv.n_pages) {
        if (err && t < t1) atomicExch(err, 1);
        continue;
      }
      const long long rowi = ((long long)page * Hkv + kvh) * kv.page_size + t % kv.page_size;
      dec_cp_async16(dk, (const uint8_t*)kv.k_pool + rowi * ROWB + part * 16);
      dec_cp_async16(dv, (const uint8_t*)kv.v_pool + rowi * ROWB + part * 16);
    }
    if constexpr (KVQ == FP_KV_INT8) {
      for (int j = tid; j < TT; j += 128) {
        const int t = tt0 + j, lp = t / kv.page_size;
        if (lp >= kv.pages_per_seq) continue;
        const int page = pt[lp];
        if (page < 0 || page >= kv.n_pages) continue;
        const long long rowi = ((long long)page * Hkv + kvh) * kv.page_size + t % kv.page_size;
        dec_cp_async4(sKs + (tile % NBUF) * TT + j, kv.k_scale + rowi);
        dec_cp_async4(sVs + (tile % NBUF) * TT + j, kv.v_scale + rowi);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
#pragma unroll
  for (int i = 0; i < NBUF - 1; ++i) {
    if (i < ntile) issue(i);
    else asm volatile("cp.async.commit_group;" ::: "memory");
  }

  // q of the G heads, this lane's dims, pre-scaled by log2(e) / sqrt(hd)
  const float qscale = kLog2e * rsqrtf((float)HD);
  float qr[G][DPL];
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int d = 0; d < DPL; ++d)
      qr[g][d] = bf2f(q[(long long)b * q_stride + (long long)(kvh * G + g) * HD + lane * DPL + d]) * qscale;
  float m[G], l[G], acc[G][DPL];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
#pragma unroll
    for (int d = 0; d < DPL; ++d) acc[g][d] = 0.f;
  }

  for (int tile = 0; tile < ntile; ++tile) {
    asm volatile("cp.async.wait_group %0;" ::"n"(NBUF - 2) : "memory");
    __syncthreads();  // tile landed for every thread; the slot refilled below is free
    if (tile + NBUF - 1 < ntile) issue(tile + NBUF - 1);
    else asm volatile("cp.async.commit_group;" ::: "memory");
    const int slot = tile % NBUF;
    const uint8_t* tK = sK + slot * TILEB;
    const uint8_t* tV = sV + slot * TILEB;
    const int tt0 = t0 + tile * TT;
#pragma unroll
    for (int grp = 0; grp < 8 / TG; ++grp) {
      float sc[TG][G];
#pragma unroll
      for (int i = 0; i < TG; ++i) {
        const int j = warp * 8 + grp * TG + i;
        if (tt0 + j < t1) {  // warp-uniform
          float kf[DPL];
          if constexpr (KVQ == FP_KV_BF16) {
            if constexpr (DPL == 4) {
              const uint2 raw = *reinterpret_cast<const uint2*>(tK + j * ROWB + lane * 8);
              const float2 a = bf2x2f(raw.x), c = bf2x2f(raw.y);
              kf[0] = a.x; kf[1] = a.y; kf[2] = c.x; kf[3] = c.y;
            } else {
              const float2 a = bf2x2f(*reinterpret_cast<const uint32_t*>(tK + j * ROWB + lane * 4));
              kf[0] = a.x; kf[1] = a.y;
            }
          } else {
            uint32_t raw;
            if constexpr (DPL == 4) raw = *reinterpret_cast<const uint32_t*>(tK + j * ROWB + lane * 4);
            else raw = *reinterpret_cast<const uint16_t*>(tK + j * ROWB + lane * 2);
#pragma unroll
            for (int d = 0; d < DPL; ++d) kf[d] = (float)(int8_t)((raw >> (8 * d)) & 0xFF);
          }
          const float ks = KVQ == FP_KV_INT8 ? sKs[slot * TT + j] : 1.f;
#pragma unroll
          for (int g = 0; g < G; ++g) {
            float a = 0.f;
#pragma unroll
            for (int d = 0; d < DPL; ++d) a += qr[g][d] * kf[d];
            sc[i][g] = warp_sum(a) * ks;
          }
        } else {
#pragma unroll
          for (int g = 0; g < G; ++g) sc[i][g] = -INFINITY;
        }
      }
      // online softmax over these TG tokens
      float p[TG][G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float mx = m[g];
#pragma unroll
        for (int i = 0; i < TG; ++i) mx = fmaxf(mx, sc[i][g]);
        const float ref = mx == -INFINITY ? 0.f : mx;
        const float corr = exp2f(m[g] - ref);
        float ps = 0.f;
#pragma unroll
        for (int i = 0; i < TG; ++i) {
          p[i][g] = exp2f(sc[i][g] - ref);
          ps += p[i][g];
        }
        l[g] = l[g] * corr + ps;
        m[g] = mx;
#pragma unroll
        for (int d = 0; d < DPL; ++d) acc[g][d] *= corr;
      }
#pragma unroll
      for (int i = 0; i < TG; ++i) {
        const int j = warp * 8 + grp * TG + i;
        if (tt0 + j < t1) {
          float vf[DPL];
          if constexpr (KVQ == FP_KV_BF16) {
            if constexpr (DPL == 4) {
              const uint2 raw = *reinterpret_cast<const uint2*>(tV + j * ROWB + lane * 8);
              const float2 a = bf2x2f(raw.x), c = bf2x2f(raw.y);
              vf[0] = a.x; vf[1] = a.y; vf[2] = c.x; vf[3] = c.y;
            } else {
              const float2 a = bf2x2f(*reinterpret_cast<const uint32_t*>(tV + j * ROWB + lane * 4));
              vf[0] = a.x; vf[1] = a.y;
            }
          } else {
            uint32_t raw;
            if constexpr (DPL == 4) raw = *reinterpret_cast<const uint32_t*>(tV + j * ROWB + lane * 4);
            else raw = *reinterpret_cast<const uint16_t*>(tV + j * ROWB + lane * 2);
            const float vs = sVs[slot * TT + j];
#pragma unroll
            for (int d = 0; d < DPL; ++d) vf[d] = (float)(int8_t)((raw >> (8 * d)) & 0xFF) * vs;
          }
#pragma unroll
          for (int g = 0; g < G; ++g)
#pragma unroll
            for (int d = 0; d < DPL; ++d) acc[g][d] += p[i][g] * vf[d];
        }
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();  // the ring is reused for the merge below

  // ---- merge the 4 warps: per head, o = sum_w acc_w 2^(m_w - M), l = sum_w l_w 2^(m_w - M)
  float* red = reinterpret_cast<float*>(smem);  // [4][G][HD + 2]
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float* r = red + (warp * G + g) * (HD + 2);
#pragma unroll
    for (int d = 0; d < DPL; ++d) r[lane * DPL + d] = acc[g][d];
    if (lane == 0) {
      r[HD] = m[g];
      r[HD + 1] = l[g];
    }
  }
  __syncthreads();
  for (int i = tid; i < G * HD; i += 128) {
    const int g = i / HD, e = i % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, red[(w * G + g) * (HD + 2) + HD]);
    float o = 0.f, L = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float* r = red + (w * G + g) * (HD + 2);
      const float f = r[HD] == -INFINITY ? 0.f : exp2f(r[HD] - M);
      o += r[e] * f;
      L += r[HD + 1] * f;
    }
    const long long row = ((long long)b * H + kvh * G + g) * splits + split;
    float* w = ws + row * (HD + 2);
    w[e] = o;
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

template <int HD, int KVQ, int G>
static cudaError_t launch_decode_t(const uint16_t* q, int q_stride, int B, int H, const fp_kv_view& kv,
                                   const int32_t* len, int len_add, int max_len, DecodeGeom g, float* ws,
                                   uint16_t* out, int32_t* err, cudaStream_t s, cudaError_t* second) {
  // the ring also holds the 4-warp merge buffer after the loop
  const size_t smem = std::max(dec_smem_bytes<HD, KVQ>(), (size_t)4 * G * (HD + 2) * sizeof(float));
  auto kern = attn_decode_kernel<HD, KVQ, G>;
  if (smem > 48 * 1024) FP_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  dim3 grid(B * kv.n_kv_heads, g.splits);
  cudaError_t e = launch(kern, grid, dim3(128), smem, s, q, q_stride, H, kv, len, len_add, max_len, g.chunk,
                         g.splits, ws, err);
  if (e != cudaSuccess) return e;
  e = launch(attn_combine_kernel<HD>, dim3(B * H), dim3(HD), 0, s, H, len, len_add, max_len, g.chunk, g.splits,
             (const float*)ws, out);
  if (second) *second = e;
  return e;
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
  DecodeGeom g = decode_geom(B, kv.n_kv_heads, max_len);
  const int G = n_heads / kv.n_kv_heads;
  float* w = (float*)ws;
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
// key/value tiles of 64 staged in shared memory as bf16; S = Q K^T and
// O += P V with mma.sync m16n8k16 (bf16 in, fp32 accumulate) and an online
// softmax in the log2 domain.
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

template <int HD, int KVQ>
__global__ void __launch_bounds__(128) attn_prefill_kernel(const uint16_t* __restrict__ q, int q_stride, int S,
                                                           int H, fp_kv_view kv, uint16_t* __restrict__ out,
                                                           int32_t* err) {
  constexpr int BT = 64;        // rows per tile
  constexpr int LD = HD + 8;    // padded row (bf16 elements) against ldmatrix bank conflicts
  extern __shared__ __align__(16) uint8_t smem_raw[];
  pdl_trigger();
  pdl_wait();
  uint16_t* sQ = reinterpret_cast<uint16_t*>(smem_raw);
  uint16_t* sK = sQ + BT * LD;
  uint16_t* sV = sK + BT * LD;
  float* sks = reinterpret_cast<float*>(sV + BT * LD);  // [BT] key scales (int8)
  float* svs = sks + BT;                                // [BT] value scales (int8)

  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int Hkv = kv.n_kv_heads, G = H / Hkv, kvh = h / G;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g8 = lane >> 2, t4 = lane & 3;
  const int q0 = qt * BT;
  constexpr int CPR = HD / 8;  // 16-byte chunks per bf16 row

  // ---- Q tile
  for (int c = tid; c < BT * CPR; c += 128) {
    const int r = c / CPR, cc = c % CPR;
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
  const int32_t* pt = kv.page_table + (long long)b * kv.pages_per_seq;
  const int last_key = min(q0 + BT, S) - 1;
  const int qrow0 = q0 + warp * 16 + g8;  // rows qrow0 and qrow0 + 8

  for (int k0 = 0; k0 <= last_key; k0 += BT) {
    __syncthreads();
    // ---- stage K and V rows k0 .. k0+63 (zeros past S)
    if (KVQ == FP_KV_BF16) {
      for (int c = tid; c < 2 * BT * CPR; c += 128) {
        const int which = c / (BT * CPR), r = (c % (BT * CPR)) / CPR, cc = c % CPR;
        const int t = k0 + r;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (t < S) {
          const int page = pt[t / kv.page_size];
          if (page >= 0 && page < kv.n_pages) {
            const long long rowi = ((long long)page * Hkv + kvh) * kv.page_size + t % kv.page_size;
            v = ld_nc16((const uint16_t*)(which ? kv.v_pool : kv.k_pool) + rowi * HD + cc * 8);
          } else if (err) {
            atomicExch(err, 1);
          }
        }
        *reinterpret_cast<uint4*>((which ? sV : sK) + r * LD + cc * 8) = v;
      }
    } else {
      constexpr int CPR8 = HD / 16;  // 16-byte chunks per int8 row
      for (int c = tid; c < 2 * BT * CPR8; c += 128) {
        const int which = c / (BT * CPR8), r = (c % (BT * CPR8)) / CPR8, cc = c % CPR8;
        const int t = k0 + r;
        uint4 v = make_uint4(0, 0, 0, 0);
        float sc = 0.f;
        if (t < S) {
          const int page = pt[t / kv.page_size];
          if (page >= 0 && page < kv.n_pages) {
            const long long rowi = ((long long)page * Hkv + kvh) * kv.page_size + t % kv.page_size;
            v = ld_nc16((const int8_t*)(which ? kv.v_pool : kv.k_pool) + rowi * HD + cc * 16);
            sc = (which ? kv.v_scale : kv.k_scale)[rowi];
          } else if (err) {
            atomicExch(err, 1);
          }
        }
        uint32_t w[4] = {v.x, v.y, v.z, v.w}, o8[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const uint32_t word = w[i >> 1];
          const int sh = 16 * (i & 1);
          const float a = (float)(int8_t)((word >> sh) & 0xFF), bb = (float)(int8_t)((word >> (sh + 8)) & 0xFF);
          o8[i] = pack_bf2(a, bb);  // small integers: exact in bf16
        }
        uint16_t* dst = (which ? sV : sK) + r * LD + cc * 16;
        *reinterpret_cast<uint4*>(dst) = make_uint4(o8[0], o8[1], o8[2], o8[3]);
        *reinterpret_cast<uint4*>(dst + 8) = make_uint4(o8[4], o8[5], o8[6], o8[7]);
        if (cc == 0) (which ? svs : sks)[r] = sc;
      }
    }
    __syncthreads();
    // ---- S = Q K^T for this warp's 16 rows x 64 keys
    float sacc[BT / 8][4];
#pragma unroll
    for (int n = 0; n < BT / 8; ++n) sacc[n][0] = sacc[n][1] = sacc[n][2] = sacc[n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int n = 0; n < BT / 8; ++n) {
        uint32_t b0, b1;
        const int r = n * 8 + (lane & 7), c = kk * 16 + 8 * ((lane >> 3) & 1);
        ldsm_x2(b0, b1, sK + r * LD + c);
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
        if (KVQ == FP_KV_INT8) v *= sks[n * 8 + 2 * t4 + (i & 1)];
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
        if (KVQ == FP_KV_INT8) p[i] *= svs[n * 8 + 2 * t4 + (i & 1)];
      }
      pa[n >> 1][(n & 1) * 2 + 0] = pack_bf2(p[0], p[1]);
      pa[n >> 1][(n & 1) * 2 + 1] = pack_bf2(p[2], p[3]);
    }
    // ---- O += P V
#pragma unroll
    for (int j = 0; j < BT / 16; ++j) {
#pragma unroll
      for (int dt = 0; dt < HD / 8; ++dt) {
        uint32_t b0, b1;
        const int r = j * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
        ldsm_x2_trans(b0, b1, sV + r * LD + dt * 8);
        mma_bf16(o[dt], pa[j], b0, b1);
      }
    }
  }
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
  constexpr int LD = HD + 8;
  size_t smem = 3 * 64 * LD * 2 + 2 * 64 * sizeof(float);
  auto kern = attn_prefill_kernel<HD, KVQ>;
  if (smem > 48 * 1024) FP_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  dim3 grid((S + 63) / 64, H, B);
  return launch(kern, grid, dim3(128), smem, s, q, q_stride, S, H, kv, out, err);
}

cudaError_t launch_attention_prefill(const uint16_t* q, int q_stride, int B, int S, int n_heads,
                                     const fp_kv_view& kv, uint16_t* out, int32_t* err, cudaStream_t s) {
  if (B <= 0 || S <= 0) return cudaSuccess;
  if (kv.head_dim == 64)
    return kv.kvquant == FP_KV_BF16 ? launch_prefill_t<64, FP_KV_BF16>(q, q_stride, B, S, n_heads, kv, out, err, s)
                                    : launch_prefill_t<64, FP_KV_INT8>(q, q_stride, B, S, n_heads, kv, out, err, s);
  return kv.kvquant == FP_KV_BF16 ? launch_prefill_t<128, FP_KV_BF16>(q, q_stride, B, S, n_heads, kv, out, err, s)
                                  : launch_prefill_t<128, FP_KV_INT8>(q, q_stride, B, S, n_heads, kv, out, err, s);
}

}  // namespace fpk
