// Device helpers shared by the decode kernels: chunked dot products over 16-byte weight chunks
// (fp32, bf16, int4 g128), streaming / L2-coherent loads, warp reductions and shared-memory
// staging. Every kernel that uses them assigns chunk c = j * 32 + lane to a lane and reduces
// with the same butterfly, so a row's result does not depend on which kernel computed it.
#pragma once
#include <cuda_bf16.h>
#include <stdint.h>

#include "kernels.cuh"

namespace moe {
namespace dev {

constexpr unsigned kFull = 0xffffffffu;

// Elements per 16-byte weight chunk, and bytes of activation that match one chunk.
template <int WD>
struct Tr;
template <>
struct Tr<WD_FP32> {
  static constexpr int epc = 4;
  static constexpr int xbytes = 16;  // 4 fp32 activations
};
template <>
struct Tr<WD_BF16> {
  static constexpr int epc = 8;
  static constexpr int xbytes = 16;  // 8 bf16 activations
};
template <>
struct Tr<WD_INT4> {
  static constexpr int epc = 32;
  static constexpr int xbytes = 64;  // 32 bf16 activations
};

__device__ __forceinline__ uint4 ld_stream(const uint8_t* p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

__device__ __forceinline__ float bf16_bits(uint32_t b) { return __uint_as_float(b << 16); }
__device__ __forceinline__ float lo_bf16(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float hi_bf16(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
  return v;
}

// acc + sum_e w_e * x_e over one 16-byte weight chunk; x points at the matching activations
// in shared memory (fp32 for fp32 weights, bf16 otherwise). int4 returns the unscaled sum of
// q_e * x_e (the group scale is applied by the caller).
template <int WD>
__device__ __forceinline__ float dot_chunk(const uint4& w, const uint8_t* x, float acc);

template <>
__device__ __forceinline__ float dot_chunk<WD_FP32>(const uint4& w, const uint8_t* x, float acc) {
  const float4 xv = *reinterpret_cast<const float4*>(x);
  acc = fmaf(__uint_as_float(w.x), xv.x, acc);
  acc = fmaf(__uint_as_float(w.y), xv.y, acc);
  acc = fmaf(__uint_as_float(w.z), xv.z, acc);
  acc = fmaf(__uint_as_float(w.w), xv.w, acc);
  return acc;
}

template <>
__device__ __forceinline__ float dot_chunk<WD_BF16>(const uint4& w, const uint8_t* x, float acc) {
  const uint4 xv = *reinterpret_cast<const uint4*>(x);
  const uint32_t wq[4] = {w.x, w.y, w.z, w.w};
  const uint32_t xq[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
  for (int k = 0; k < 4; k++) {
    acc = fmaf(lo_bf16(wq[k]), lo_bf16(xq[k]), acc);
    acc = fmaf(hi_bf16(wq[k]), hi_bf16(xq[k]), acc);
  }
  return acc;
}

// Nibble p of 32-bit word k is element 8k + p. With the word xor 0x88888888 each nibble n is
// q + 8 in [0, 15]; 0x4B000000 | n is the float 2^23 + n exactly, so subtracting 2^23 + 8
// yields q exactly.
template <>
__device__ __forceinline__ float dot_chunk<WD_INT4>(const uint4& w, const uint8_t* x, float acc) {
  const uint32_t wq[4] = {w.x ^ 0x88888888u, w.y ^ 0x88888888u, w.z ^ 0x88888888u, w.w ^ 0x88888888u};
#pragma unroll
  for (int k = 0; k < 4; k++) {
    const uint4 xv = *reinterpret_cast<const uint4*>(x + 16 * k);  // 8 bf16 activations
    const uint32_t xq[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
    for (int p = 0; p < 8; p++) {
      const float q = __uint_as_float(0x4B000000u | ((wq[k] >> (4 * p)) & 0xFu)) - 8388616.0f;
      const float xe = (p & 1) ? hi_bf16(xq[p >> 1]) : lo_bf16(xq[p >> 1]);
      acc = fmaf(q, xe, acc);
    }
  }
  return acc;
}

// Copy nbytes (a multiple of 16) from global to shared memory with 16-byte loads.
__device__ __forceinline__ void stage16(uint4* dst, const void* src, int nbytes, int tid, int nthreads) {
  const uint4* s = reinterpret_cast<const uint4*>(src);
  const int n = nbytes >> 4;
#pragma unroll 4
  for (int c = tid; c < n; c += nthreads) dst[c] = __ldg(s + c);
}

// Order-preserving map of a float to uint32 (larger float -> larger key; -0 treated as +0).
__device__ __forceinline__ uint32_t ord_key(float f) {
  uint32_t u = __float_as_uint(f == 0.0f ? 0.0f : f);
  const uint32_t key = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  // key 0 is reserved: the top-k selections use it for "taken or absent". The one float that
  // would map to it, the negative NaN with every bit set, takes key 1 and sorts with the other
  // negative NaNs, below -inf.
  return key > 1u ? key : 1u;
}
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

__device__ __forceinline__ uint4 ld_cg(const uint8_t* p) {
  uint4 r;
  asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ void st_v4(uint8_t* p, const uint4& v) {
  asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}

// An empty asm that claims to rewrite w: a loop that applies the same packed weights to several
// activation vectors then unpacks them inside the loop instead of keeping every unpacked value
// live across it (which would not fit in registers).
__device__ __forceinline__ void opaque(uint4& w) {
  asm volatile("" : "+r"(w.x), "+r"(w.y), "+r"(w.z), "+r"(w.w));
}

__host__ __device__ __forceinline__ int upad(int i) { return i + 4 * (i >> 5); }
__host__ __device__ __forceinline__ int ipad_of(int I) { return upad((I + 31) & ~31); }

template <int WD>
__device__ __forceinline__ float dot_chunk_u(const uint4& w, const float* u, float acc);

template <>
__device__ __forceinline__ float dot_chunk_u<WD_FP32>(const uint4& w, const float* u, float acc) {
  const float4 v = *reinterpret_cast<const float4*>(u);
  acc = fmaf(__uint_as_float(w.x), v.x, acc);
  acc = fmaf(__uint_as_float(w.y), v.y, acc);
  acc = fmaf(__uint_as_float(w.z), v.z, acc);
  acc = fmaf(__uint_as_float(w.w), v.w, acc);
  return acc;
}

template <>
__device__ __forceinline__ float dot_chunk_u<WD_BF16>(const uint4& w, const float* u, float acc) {
  const float4 v0 = *reinterpret_cast<const float4*>(u);
  const float4 v1 = *reinterpret_cast<const float4*>(u + 4);
  acc = fmaf(lo_bf16(w.x), v0.x, acc);
  acc = fmaf(hi_bf16(w.x), v0.y, acc);
  acc = fmaf(lo_bf16(w.y), v0.z, acc);
  acc = fmaf(hi_bf16(w.y), v0.w, acc);
  acc = fmaf(lo_bf16(w.z), v1.x, acc);
  acc = fmaf(hi_bf16(w.z), v1.y, acc);
  acc = fmaf(lo_bf16(w.w), v1.z, acc);
  acc = fmaf(hi_bf16(w.w), v1.w, acc);
  return acc;
}

template <>
__device__ __forceinline__ float dot_chunk_u<WD_INT4>(const uint4& w, const float* u, float acc) {
  const uint32_t wq[4] = {w.x ^ 0x88888888u, w.y ^ 0x88888888u, w.z ^ 0x88888888u, w.w ^ 0x88888888u};
#pragma unroll
  for (int k = 0; k < 4; k++) {
    const float4 v0 = *reinterpret_cast<const float4*>(u + 8 * k);
    const float4 v1 = *reinterpret_cast<const float4*>(u + 8 * k + 4);
    const float uv[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
    for (int p = 0; p < 8; p++) {
      const float q = __uint_as_float(0x4B000000u | ((wq[k] >> (4 * p)) & 0xFu)) - 8388616.0f;
      acc = fmaf(q, uv[p], acc);
    }
  }
  return acc;
}

}  // namespace dev
}  // namespace moe
