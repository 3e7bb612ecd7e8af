// Row-wise kernels of the fingerprint block: embedding gather (alone or fused
// with the first RMSNorm), RMSNorm, RoPE + KV-cache append (with the int8 KV
// quantiser fused into the cache write) and greedy argmax (optionally
// advancing the position counter).
//
// Components: embedding, normalisation and the LM head's greedy choice are
// among the fingerprint's components (Sec. 1 "Our work"; Sec. 5.1); the KV
// cache and its INT8 variant are a deployment configuration (Sec. 2, Sec. 3.2,
// table "Models and configurations"); the KV cache keeps per-token decode
// cost constant (Sec. 5.3, before Eq. 1).
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.cuh"

namespace cg = cooperative_groups;

namespace fpk {

// ------------------------------------------------------------------ embedding
// One CTA per token row; 16-byte copies (d % 8 == 0).
__global__ void embed_kernel(const int32_t* __restrict__ tok, const uint16_t* __restrict__ E, int V, int d,
                             uint16_t* __restrict__ h, int32_t* err) {
  pdl_trigger();
  pdl_wait();
  const long long m = blockIdx.x;
  int t = tok[m];
  uint4* dst = reinterpret_cast<uint4*>(h + m * d);
  const int chunks = d / 8;
  if (t < 0 || t >= V) {
    if (threadIdx.x == 0 && err) atomicExch(err, 1);
    for (int c = threadIdx.x; c < chunks; c += blockDim.x) dst[c] = make_uint4(0, 0, 0, 0);
    return;
  }
  const uint4* src = reinterpret_cast<const uint4*>(E + (long long)t * d);
  for (int c = threadIdx.x; c < chunks; c += blockDim.x) dst[c] = ld_nc16(src + c);
}

cudaError_t launch_embed(const int32_t* tok, int M, const uint16_t* E, int V, int d, uint16_t* h, int32_t* err,
                         cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  return launch(embed_kernel, dim3(M), dim3(128), 0, s, tok, E, V, d, h, err);
}

// ------------------------------------------------------------------ embedding + RMSNorm
// The embedding gather fused with the first block's pre-attention RMSNorm:
// one CTA of 128 threads per token row writes h = E[tok] and
// y = h * rsqrt(mean(h^2) + eps) * g (fp32 math), as embed_kernel followed
// by rmsnorm_kernel would.  An out-of-range id gives h = y = 0 and err = 1.
__global__ void embed_rmsnorm_kernel(const int32_t* __restrict__ tok, const uint16_t* __restrict__ E, int V, int d,
                                     uint16_t* __restrict__ h, const uint16_t* __restrict__ g, float eps,
                                     uint16_t* __restrict__ y, int32_t* err) {
  pdl_trigger();
  pdl_wait();
  const long long m = blockIdx.x;
  const int t = tok[m];
  uint4* hr = reinterpret_cast<uint4*>(h + m * d);
  uint4* yr = reinterpret_cast<uint4*>(y + m * d);
  const int chunks = d / 8;
  if (t < 0 || t >= V) {
    if (threadIdx.x == 0 && err) atomicExch(err, 1);
    for (int c = threadIdx.x; c < chunks; c += blockDim.x) hr[c] = yr[c] = make_uint4(0, 0, 0, 0);
    return;
  }
  const uint4* src = reinterpret_cast<const uint4*>(E + (long long)t * d);
  const uint4* gr = reinterpret_cast<const uint4*>(g);
  float ss = 0.f;
  for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
    const uint4 v = ld_nc16(src + c);
    hr[c] = v;
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = bf2x2f(w[i]);
      ss += f.x * f.x + f.y * f.y;
    }
  }
  ss = warp_sum(ss);
  __shared__ float red[4];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  const float inv = rsqrtf((red[0] + red[1] + red[2] + red[3]) / (float)d + eps);
  for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
    const uint4 v = ld_nc16(src + c), gg = gr[c];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w}, gw[4] = {gg.x, gg.y, gg.z, gg.w};
    uint32_t o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = bf2x2f(w[i]), gf = bf2x2f(gw[i]);
      o[i] = pack_bf2(f.x * inv * gf.x, f.y * inv * gf.y);
    }
    yr[c] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

cudaError_t launch_embed_rmsnorm(const int32_t* tok, int M, const uint16_t* E, int V, int d, uint16_t* h,
                                 const uint16_t* g, float eps, uint16_t* y, int32_t* err, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  return launch(embed_rmsnorm_kernel, dim3(M), dim3(128), 0, s, tok, E, V, d, h, g, eps, y, err);
}

// ------------------------------------------------------------------ RMSNorm
// y[r] = x[r * stride + offset] * rsqrt(mean(x^2) + eps) * g, fp32 math.
// One CTA of 128 threads per row; 16-byte loads (d % 8 == 0).
__global__ void rmsnorm_kernel(const uint16_t* __restrict__ x, int d, int row_stride, int row_offset,
                               const uint16_t* __restrict__ g, float eps, uint16_t* __restrict__ y) {
  pdl_trigger();
  pdl_wait();
  const long long r = blockIdx.x;
  const uint4* xr = reinterpret_cast<const uint4*>(x + ((long long)r * row_stride + row_offset) * d);
  const uint4* gr = reinterpret_cast<const uint4*>(g);
  uint4* yr = reinterpret_cast<uint4*>(y + r * d);
  const int chunks = d / 8;
  float ss = 0.f;
  for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
    uint4 v = xr[c];
    uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 f = bf2x2f(w[i]);
      ss += f.x * f.x + f.y * f.y;
    }
  }
  ss = warp_sum(ss);
  __shared__ float red[4];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = red[0] + red[1] + red[2] + red[3];
  float inv = rsqrtf(tot / (float)d + eps);
  for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
    uint4 v = xr[c], gg = gr[c];
    uint32_t w[4] = {v.x, v.y, v.z, v.w}, gw[4] = {gg.x, gg.y, gg.z, gg.w}, o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 f = bf2x2f(w[i]), gf = bf2x2f(gw[i]);
      o[i] = pack_bf2(f.x * inv * gf.x, f.y * inv * gf.y);
    }
    yr[c] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

cudaError_t launch_rmsnorm(const uint16_t* x, int M, int d, int row_stride, int row_offset, const uint16_t* g,
                           float eps, uint16_t* y, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  return launch(rmsnorm_kernel, dim3(M), dim3(128), 0, s, x, d, row_stride, row_offset, g, eps, y);
}

// ------------------------------------------------------------------ argmax
// A cluster of kArgmaxCTAs CTAs per row: each CTA finds the first maximum of
// its slice, then CTA 0 of the cluster reads the slices' winners from the
// other CTAs' shared memory (distributed shared memory) and keeps the first
// maximum.  Ties go to the lowest index.
constexpr int kArgmaxCTAs = 8;

FP_DEV void better(float& bv, int& bi, float v, int i) {
  if (v > bv || (v == bv && i < bi)) {
    bv = v;
    bi = i;
  }
}

__global__ void __cluster_dims__(kArgmaxCTAs, 1, 1) __launch_bounds__(256)
    argmax_kernel(const float* __restrict__ logits, int V, int32_t* __restrict__ out, int32_t* pos, int by) {
  __shared__ float sv[8];
  __shared__ int si[8];
  __shared__ float cv;
  __shared__ int ci;
  pdl_trigger();
  pdl_wait();
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int row = blockIdx.y;
  const float* lr = logits + (long long)row * V;
  // slices start on multiples of 4 so rows whose start is 16-byte aligned read float4s
  const int per = ((V + kArgmaxCTAs - 1) / kArgmaxCTAs + 3) & ~3;
  const int lo = min(V, rank * per), hi = min(V, lo + per);
  float best = -INFINITY;
  int bi = 0x7fffffff;
  if ((V & 3) == 0 && ((uintptr_t)lr & 15) == 0) {
    const float4* l4 = reinterpret_cast<const float4*>(lr);
#pragma unroll 4
    for (int i = (lo >> 2) + (int)threadIdx.x; i < (hi >> 2); i += blockDim.x) {
      const float4 v = __ldg(l4 + i);
      better(best, bi, v.x, 4 * i);
      better(best, bi, v.y, 4 * i + 1);
      better(best, bi, v.z, 4 * i + 2);
      better(best, bi, v.w, 4 * i + 3);
    }
  } else {
    for (int i = lo + (int)threadIdx.x; i < hi; i += blockDim.x) better(best, bi, lr[i], i);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    better(best, bi, ov, oi);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    sv[warp] = best;
    si[warp] = bi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) better(best, bi, sv[w], si[w]);
    cv = best;
    ci = bi;
  }
  cluster.sync();  // every CTA's winner is in its shared memory
  if (rank == 0 && threadIdx.x == 0) {
    float b = -INFINITY;
    int i = 0x7fffffff;
    for (int r = 0; r < kArgmaxCTAs; ++r) {
      const float* rv = cluster.map_shared_rank(&cv, r);
      const int* ri = cluster.map_shared_rank(&ci, r);
      better(b, i, *rv, *ri);
    }
    out[row] = i == 0x7fffffff ? 0 : i;
    if (pos) pos[row] += by;  // the sequence's next position (the decode step is complete)
  }
  cluster.sync();  // keep the winners alive until CTA 0 has read them
}

cudaError_t launch_argmax(const float* logits, int M, int V, int32_t* out, cudaStream_t s, int32_t* pos, int by) {
  if (M <= 0) return cudaSuccess;
  return launch(argmax_kernel, dim3(kArgmaxCTAs, M), dim3(256), 0, s, logits, V, out, pos, by);
}

// ------------------------------------------------------------------ RoPE + KV append
// One warp per (token, head slot); slots are the H query heads, then the Hkv
// key heads, then the Hkv value heads.  Lane l holds elements l + 32 j, so
// each rotate-half pair (i, i + hd/2) sits in one lane.  Rotation in fp32,
// rounded to bf16.  Keys and values go to the paged cache; with an int8
// cache each (token, KV head) row is quantised: s = fp32(max|x| / 127),
// q = clamp(rint(fp32(x / s)), -127, 127).
//
// No early trigger: the attention after it is launched once this kernel has
// finished, when the linear before it has left every SM, so that its CTAs
// spread over all SMs (launched early, they piled up on the first SMs the
// linear freed).
template <int HD, int KVQ>
__global__ void rope_kv_kernel(uint16_t* __restrict__ qkv, int B, int S, int row_stride, int H, fp_kv_view kv,
                               const int32_t* __restrict__ pos, const float* __restrict__ cs, int32_t* err) {
  pdl_wait();
  constexpr int E = HD / 32;
  const int Hkv = kv.n_kv_heads;
  const int slots = H + 2 * Hkv;
  const long long wid = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (wid >= (long long)B * S * slots) return;
  const int lane = threadIdx.x & 31;
  const int slot = (int)(wid % slots);
  const long long m = wid / slots;
  const int b = (int)(m / S), s = (int)(m % S);
  const int p = pos[b] + s;
  const int lp = p / kv.page_size;
  if (p < 0 || lp >= kv.pages_per_seq) {  // outside the cache and the RoPE table: skip
    if (lane == 0 && err) atomicExch(err, 1);
    return;
  }
  uint16_t* src = qkv + m * row_stride + (long long)slot * HD;  // q | k | v heads are contiguous
  float x[E];
#pragma unroll
  for (int j = 0; j < E; ++j) x[j] = bf2f(src[lane + 32 * j]);
  const bool is_v = slot >= H + Hkv;
  if (!is_v) {
    const float* c = cs + (long long)p * HD;  // [p][HD/2][2]
#pragma unroll
    for (int j = 0; j < E / 2; ++j) {
      const int i = lane + 32 * j;
      const float co = c[2 * i], si = c[2 * i + 1];
      const float a = x[j], bb = x[j + E / 2];
      x[j] = a * co - bb * si;
      x[j + E / 2] = bb * co + a * si;
    }
#pragma unroll
    for (int j = 0; j < E; ++j) x[j] = bf2f(f2bf(x[j]));
  }
  if (slot < H) {
#pragma unroll
    for (int j = 0; j < E; ++j) src[lane + 32 * j] = f2bf(x[j]);
    return;
  }
  const int kvh = is_v ? slot - H - Hkv : slot - H;
  const int page = kv.page_table[(long long)b * kv.pages_per_seq + lp];
  if (page < 0 || page >= kv.n_pages) {
    if (lane == 0 && err) atomicExch(err, 1);
    return;
  }
  const long long rowi = ((long long)page * Hkv + kvh) * kv.page_size + (p % kv.page_size);
  if (KVQ == FP_KV_BF16) {
    uint16_t* dst = (uint16_t*)(is_v ? kv.v_pool : kv.k_pool) + rowi * HD;
#pragma unroll
    for (int j = 0; j < E; ++j) dst[lane + 32 * j] = f2bf(x[j]);
  } else {
    float amax = 0.f;
#pragma unroll
    for (int j = 0; j < E; ++j) amax = fmaxf(amax, fabsf(x[j]));
    amax = warp_max(amax);
    const float sc = __fdiv_rn(amax, 127.0f);
    int8_t* dst = (int8_t*)(is_v ? kv.v_pool : kv.k_pool) + rowi * HD;
#pragma unroll
    for (int j = 0; j < E; ++j) {
      float r = sc > 0.f ? rintf(__fdiv_rn(x[j], sc)) : 0.f;
      dst[lane + 32 * j] = (int8_t)(int)fminf(fmaxf(r, -127.f), 127.f);
    }
    if (lane == 0) (is_v ? kv.v_scale : kv.k_scale)[rowi] = sc;
  }
}

cudaError_t launch_rope_kv(uint16_t* qkv, int B, int S, int row_stride, int n_heads, const fp_kv_view& kv,
                           const int32_t* pos, const float* rope_cs, int32_t* err, cudaStream_t s) {
  long long warps = (long long)B * S * (n_heads + 2 * kv.n_kv_heads);
  if (warps <= 0) return cudaSuccess;
  int blocks = (int)((warps + 7) / 8);
  if (kv.head_dim == 64) {
    if (kv.kvquant == FP_KV_BF16)
      return launch(rope_kv_kernel<64, FP_KV_BF16>, dim3(blocks), dim3(256), 0, s, qkv, B, S, row_stride, n_heads, kv, pos, rope_cs, err);
    else
      return launch(rope_kv_kernel<64, FP_KV_INT8>, dim3(blocks), dim3(256), 0, s, qkv, B, S, row_stride, n_heads, kv, pos, rope_cs, err);
  } else {
    if (kv.kvquant == FP_KV_BF16)
      return launch(rope_kv_kernel<128, FP_KV_BF16>, dim3(blocks), dim3(256), 0, s, qkv, B, S, row_stride, n_heads, kv, pos, rope_cs, err);
    else
      return launch(rope_kv_kernel<128, FP_KV_INT8>, dim3(blocks), dim3(256), 0, s, qkv, B, S, row_stride, n_heads, kv, pos, rope_cs, err);
  }
  return cudaGetLastError();
}

}  // namespace fpk
