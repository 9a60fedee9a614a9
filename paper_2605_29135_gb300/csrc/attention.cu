// Grouped-query attention of one decode token over a KV cache: the attention of the decoder block
// around the MoE layer (a stack decoded at a 4096-token context). Flash-decoding layout: the cached
// positions of each kv head are split across CTAs; a CTA keeps, for every query head that reads the
// kv head, a running maximum, a running sum and a running weighted sum of value rows over its
// positions (each K and V row is read once for all of those heads), and a second kernel merges the
// splits with their maxima.
//
// Arithmetic: fp32 throughout on bf16 or fp32 K/V and fp32 q; scores are q . k / sqrt(D) with the
// scale folded into q; exponentials by expf against the running maximum.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "moe.h"
#include "moe_internal.h"

namespace {

constexpr int kAttnWarps = 8;
constexpr unsigned kFullMask = 0xffffffffu;

__device__ __forceinline__ float warp_allsum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(kFullMask, v, off);
  return v;
}

// VPL consecutive elements of a row (VPL = 2 or 4), widened exactly to fp32.
template <int VPL>
__device__ __forceinline__ void load_row(const float* p, float (&f)[VPL]) {
  static_assert(VPL == 2 || VPL == 4, "head_dim 64 or 128");
  if constexpr (VPL == 4) {
    const float4 w = __ldg(reinterpret_cast<const float4*>(p));
    f[0] = w.x;
    f[1] = w.y;
    f[2] = w.z;
    f[3] = w.w;
  } else {
    const float2 w = __ldg(reinterpret_cast<const float2*>(p));
    f[0] = w.x;
    f[1] = w.y;
  }
}

template <int VPL>
__device__ __forceinline__ void load_row(const __nv_bfloat16* p, float (&f)[VPL]) {
  static_assert(VPL == 2 || VPL == 4, "head_dim 64 or 128");
  if constexpr (VPL == 4) {
    const uint2 w = __ldg(reinterpret_cast<const uint2*>(p));
    f[0] = __uint_as_float(w.x << 16);
    f[1] = __uint_as_float(w.x & 0xffff0000u);
    f[2] = __uint_as_float(w.y << 16);
    f[3] = __uint_as_float(w.y & 0xffff0000u);
  } else {
    const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(p));
    f[0] = __uint_as_float(w << 16);
    f[1] = __uint_as_float(w & 0xffff0000u);
  }
}

// Split sp of kv head g: positions [sp * per, min(T, (sp + 1) * per)). Warp w takes positions
// p0 + w, p0 + w + 8, ...; lane holds dims [lane * VPL, lane * VPL + VPL) of every vector. The CTA's
// warps are merged in shared memory into part[g][sp][h] = (acc[D], max, sum).
template <typename CT, int VPL, int G>
__global__ void __launch_bounds__(kAttnWarps * 32) k_attn_split(const float* q, const CT* K, const CT* V,
                                                                int64_t Tmax, int64_t T, int64_t per, int nsplit,
                                                                float* part) {
  constexpr int D = 32 * VPL;
  __shared__ float s_m[kAttnWarps][G], s_l[kAttnWarps][G];
  __shared__ float s_acc[kAttnWarps][G][D];
  const int g = blockIdx.y, sp = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float scale = rsqrtf((float)D);
  float qr[G][VPL];
#pragma unroll
  for (int h = 0; h < G; h++)
#pragma unroll
    for (int v = 0; v < VPL; v++) qr[h][v] = q[(int64_t)(g * G + h) * D + lane * VPL + v] * scale;
  float m[G], l[G], acc[G][VPL];
#pragma unroll
  for (int h = 0; h < G; h++) {
    m[h] = -INFINITY;
    l[h] = 0.f;
#pragma unroll
    for (int v = 0; v < VPL; v++) acc[h][v] = 0.f;
  }
  const int64_t p0 = (int64_t)sp * per;
  const int64_t p1 = p0 + per < T ? p0 + per : T;
  const CT* Kg = K + (int64_t)g * Tmax * D + lane * VPL;
  const CT* Vg = V + (int64_t)g * Tmax * D + lane * VPL;
  // two-stage pipeline: the next position's K and V rows are requested before this one is used
  float kf[VPL], vf[VPL], kn[VPL], vn[VPL];
  if (p0 + warp < p1) {
    load_row<VPL>(Kg + (p0 + warp) * D, kf);
    load_row<VPL>(Vg + (p0 + warp) * D, vf);
  }
  for (int64_t j = p0 + warp; j < p1; j += kAttnWarps) {
    const int64_t jn = j + kAttnWarps;
    if (jn < p1) {
      load_row<VPL>(Kg + jn * D, kn);
      load_row<VPL>(Vg + jn * D, vn);
    }
#pragma unroll
    for (int h = 0; h < G; h++) {
      float s = 0.f;
#pragma unroll
      for (int v = 0; v < VPL; v++) s = fmaf(qr[h][v], kf[v], s);
      s = warp_allsum(s);
      const float mn = fmaxf(m[h], s);
      const float c = expf(m[h] - mn);  // 0 while m is -inf
      const float p = expf(s - mn);
      l[h] = fmaf(l[h], c, p);
#pragma unroll
      for (int v = 0; v < VPL; v++) acc[h][v] = fmaf(acc[h][v], c, p * vf[v]);
      m[h] = mn;
    }
#pragma unroll
    for (int v = 0; v < VPL; v++) {
      kf[v] = kn[v];
      vf[v] = vn[v];
    }
  }
#pragma unroll
  for (int h = 0; h < G; h++) {
    if (lane == 0) {
      s_m[warp][h] = m[h];
      s_l[warp][h] = l[h];
    }
#pragma unroll
    for (int v = 0; v < VPL; v++) s_acc[warp][h][lane * VPL + v] = acc[h][v];
  }
  __syncthreads();
  // every split holds at least one position, so some warp's maximum is finite
  for (int i = threadIdx.x; i < G * D; i += blockDim.x) {
    const int h = i / D, dd = i - h * D;
    float M = -INFINITY;
    for (int w = 0; w < kAttnWarps; w++) M = fmaxf(M, s_m[w][h]);
    float L = 0.f, A = 0.f;
    for (int w = 0; w < kAttnWarps; w++) {
      if (s_m[w][h] == -INFINITY) continue;  // a warp without positions
      const float c = expf(s_m[w][h] - M);
      L = fmaf(s_l[w][h], c, L);
      A = fmaf(s_acc[w][h][dd], c, A);
    }
    float* out = part + (((int64_t)g * nsplit + sp) * G + h) * (D + 2);
    out[dd] = A;
    if (dd == 0) {
      out[D] = M;
      out[D + 1] = L;
    }
  }
}

// out[h] = sum_s acc_s exp(m_s - M) / sum_s l_s exp(m_s - M) over the splits of h's kv head; one CTA
// per query head, one thread per dim. The splits' maxima and sums are first staged in shared
// memory by all threads at once and the weights exp(m_s - M) formed once per split; each sum still
// runs over the splits in ascending order.
__global__ void k_attn_merge(const float* part, int D, int G, int nsplit, float* out) {
  extern __shared__ float s_ml[];  // [2][nsplit]: the splits' maxima, then their weights; their sums
  __shared__ float s_M, s_L;
  float* s_c = s_ml;
  float* s_l = s_ml + nsplit;
  const int h = blockIdx.x, dd = threadIdx.x;
  const int g = h / G, hh = h - g * G;
  const float* base = part + ((int64_t)g * nsplit * G + hh) * (D + 2);
  const int64_t stride = (int64_t)G * (D + 2);
  for (int sp = threadIdx.x; sp < nsplit; sp += blockDim.x) {
    s_c[sp] = base[sp * stride + D];
    s_l[sp] = base[sp * stride + D + 1];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float M = -INFINITY;
    for (int sp = 0; sp < nsplit; sp++) M = fmaxf(M, s_c[sp]);
    s_M = M;
  }
  __syncthreads();
  const float M = s_M;
  for (int sp = threadIdx.x; sp < nsplit; sp += blockDim.x) s_c[sp] = expf(s_c[sp] - M);
  __syncthreads();
  if (threadIdx.x == 0) {
    float L = 0.f;
    for (int sp = 0; sp < nsplit; sp++) L = fmaf(s_l[sp], s_c[sp], L);
    s_L = L;
  }
  float A = 0.f;
#pragma unroll 16
  for (int sp = 0; sp < nsplit; sp++) A = fmaf(base[sp * stride + dd], s_c[sp], A);
  __syncthreads();
  out[(int64_t)h * D + dd] = A / s_L;
}

// Splits per kv head: about two CTAs per SM over all kv heads, at least 16 positions each, and no
// empty split.
void split_plan(int32_t n_kv_heads, int64_t n_pos, int* nsplit, int64_t* per) {
  int64_t ns = 304 / n_kv_heads;
  if (ns < 1) ns = 1;
  const int64_t by_len = (n_pos + 15) / 16;
  if (ns > by_len) ns = by_len;
  int64_t p = (n_pos + ns - 1) / ns;
  ns = (n_pos + p - 1) / p;
  *nsplit = (int)ns;
  *per = p;
}

template <typename CT, int VPL>
cudaError_t launch_split(int G, const float* q, const CT* K, const CT* V, int Hkv, int64_t Tmax, int64_t T,
                         int64_t per, int nsplit, float* part, cudaStream_t s) {
  const dim3 grid(nsplit, Hkv), block(kAttnWarps * 32);
  switch (G) {
    case 1: k_attn_split<CT, VPL, 1><<<grid, block, 0, s>>>(q, K, V, Tmax, T, per, nsplit, part); break;
    case 2: k_attn_split<CT, VPL, 2><<<grid, block, 0, s>>>(q, K, V, Tmax, T, per, nsplit, part); break;
    case 4: k_attn_split<CT, VPL, 4><<<grid, block, 0, s>>>(q, K, V, Tmax, T, per, nsplit, part); break;
    case 8: k_attn_split<CT, VPL, 8><<<grid, block, 0, s>>>(q, K, V, Tmax, T, per, nsplit, part); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

template <typename CT>
cudaError_t launch_attention(const float* q, const void* k_cache, const void* v_cache, int32_t n_heads,
                             int32_t n_kv_heads, int32_t head_dim, int64_t max_pos, int64_t n_pos, float* out,
                             float* scratch, cudaStream_t s) {
  int nsplit;
  int64_t per;
  split_plan(n_kv_heads, n_pos, &nsplit, &per);
  const int G = n_heads / n_kv_heads;
  const CT* K = (const CT*)k_cache;
  const CT* V = (const CT*)v_cache;
  cudaError_t e = head_dim == 128 ? launch_split<CT, 4>(G, q, K, V, n_kv_heads, max_pos, n_pos, per, nsplit, scratch, s)
                                  : launch_split<CT, 2>(G, q, K, V, n_kv_heads, max_pos, n_pos, per, nsplit, scratch, s);
  if (e != cudaSuccess) return e;
  k_attn_merge<<<n_heads, head_dim, 2 * nsplit * sizeof(float), s>>>(scratch, head_dim, G, nsplit, out);
  return cudaGetLastError();
}

bool valid_shape(int32_t n_heads, int32_t n_kv_heads, int32_t head_dim) {
  if (head_dim != 64 && head_dim != 128) return false;
  if (n_kv_heads < 1 || n_heads < n_kv_heads || n_heads % n_kv_heads) return false;
  const int G = n_heads / n_kv_heads;
  return G == 1 || G == 2 || G == 4 || G == 8;
}

}  // namespace

namespace moe {

bool attention_shape_ok(int32_t n_heads, int32_t n_kv_heads, int32_t head_dim) {
  return valid_shape(n_heads, n_kv_heads, head_dim);
}

// split_plan gives at most min(304 / n_kv_heads, ceil(n_pos / 16)) splits (and at least one), a
// bound that only grows with n_pos, so this many partials serve every n_pos <= max_pos.
int64_t attention_scratch_bound(int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t max_pos) {
  int64_t ns = 304 / n_kv_heads;
  const int64_t by_len = (max_pos + 15) / 16;
  if (ns > by_len) ns = by_len;
  if (ns < 1) ns = 1;
  return (int64_t)n_heads * ns * (head_dim + 2);
}

cudaError_t attention_launch(int32_t cache_dtype, const float* q, const void* k_cache, const void* v_cache,
                             int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t max_pos, int64_t n_pos,
                             float* out, float* scratch, cudaStream_t s) {
  if (cache_dtype == MOE_DTYPE_FP32)
    return launch_attention<float>(q, k_cache, v_cache, n_heads, n_kv_heads, head_dim, max_pos, n_pos, out, scratch, s);
  return launch_attention<__nv_bfloat16>(q, k_cache, v_cache, n_heads, n_kv_heads, head_dim, max_pos, n_pos, out,
                                         scratch, s);
}

}  // namespace moe

extern "C" {

int64_t moe_attention_scratch_floats(int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t n_pos) {
  if (!valid_shape(n_heads, n_kv_heads, head_dim) || n_pos < 1) return -1;
  int nsplit;
  int64_t per;
  split_plan(n_kv_heads, n_pos, &nsplit, &per);
  return (int64_t)n_heads * nsplit * (head_dim + 2);
}

moe_status moe_attention_decode(const float* q, const void* k_cache, const void* v_cache, int32_t cache_dtype,
                                int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t max_pos, int64_t n_pos,
                                float* out, float* scratch, int64_t scratch_floats, void* stream) {
  if (!q || !k_cache || !v_cache || !out || !scratch) return MOE_ERR_INVALID;
  if (cache_dtype != MOE_DTYPE_FP32 && cache_dtype != MOE_DTYPE_BF16) return MOE_ERR_INVALID;
  if (!valid_shape(n_heads, n_kv_heads, head_dim) || n_pos < 1 || n_pos > max_pos) return MOE_ERR_INVALID;
  if (((uintptr_t)k_cache | (uintptr_t)v_cache) & 15) return MOE_ERR_INVALID;
  if (scratch_floats < moe_attention_scratch_floats(n_heads, n_kv_heads, head_dim, n_pos)) return MOE_ERR_INVALID;
  const cudaError_t e = moe::attention_launch(cache_dtype, q, k_cache, v_cache, n_heads, n_kv_heads, head_dim, max_pos,
                                              n_pos, out, scratch, (cudaStream_t)stream);
  return e == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
}

}  // extern "C"
