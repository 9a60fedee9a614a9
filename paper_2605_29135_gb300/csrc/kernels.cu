// Router / top-k, SwiGLU gate-up GEMV and down-projection + combine kernels (sm_103a).
//
// All three are HBM-bandwidth kernels at batch 1: each weight byte is read once per use with
// 128-bit streaming loads (L1 no-allocate), the input vector of a warp sits in registers
// (reused across every row the warp processes), each row's dot product is reduced with a fixed
// XOR-shuffle butterfly, and accumulation is fp32. The reduction orders do not depend on which
// slot an expert sits in or on the grid size, so results are bit-identical between capped and
// uncapped pools.
#include <cuda_bf16.h>
#include <math.h>

#include "kernels.cuh"

namespace moe {

BlobLayout make_layout(int wd, int64_t d, int64_t I) {
  BlobLayout L{};
  if (wd == WD_INT4) {
    L.row_bytes_gu = d / 2;
    L.row_bytes_d = I / 2;
    L.gu_scale_off = I * 2 * L.row_bytes_gu;
    L.d_off = L.gu_scale_off + I * 2 * (d / 128) * 2;
    L.d_scale_off = L.d_off + d * L.row_bytes_d;
    L.total = L.d_scale_off + d * (I / 128) * 2;
  } else {
    const int64_t eb = wd == WD_FP32 ? 4 : 2;
    L.row_bytes_gu = d * eb;
    L.row_bytes_d = I * eb;
    L.gu_scale_off = 0;
    L.d_off = I * 2 * L.row_bytes_gu;
    L.d_scale_off = 0;
    L.total = L.d_off + d * L.row_bytes_d;
  }
  return L;
}

namespace {

constexpr unsigned kFull = 0xffffffffu;

template <int WD>
struct Epc;  // elements per 16-byte chunk
template <>
struct Epc<WD_FP32> {
  static constexpr int v = 4;
};
template <>
struct Epc<WD_BF16> {
  static constexpr int v = 8;
};
template <>
struct Epc<WD_INT4> {
  static constexpr int v = 32;
};

__device__ __forceinline__ uint4 ld_stream(const uint8_t* p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

__device__ __forceinline__ float bf16_bits(uint32_t b) { return __uint_as_float(b << 16); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
  return v;
}

// acc + sum_e w_e * x_e over one 16-byte chunk (fp32 / bf16 storage).
template <int WD>
__device__ __forceinline__ float dot_chunk(const uint4& w, const float* x, float acc);

template <>
__device__ __forceinline__ float dot_chunk<WD_FP32>(const uint4& w, const float* x, float acc) {
  acc = fmaf(__uint_as_float(w.x), x[0], acc);
  acc = fmaf(__uint_as_float(w.y), x[1], acc);
  acc = fmaf(__uint_as_float(w.z), x[2], acc);
  acc = fmaf(__uint_as_float(w.w), x[3], acc);
  return acc;
}

template <>
__device__ __forceinline__ float dot_chunk<WD_BF16>(const uint4& w, const float* x, float acc) {
  const uint32_t q[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int k = 0; k < 4; k++) {
    acc = fmaf(__uint_as_float(q[k] << 16), x[2 * k], acc);
    acc = fmaf(__uint_as_float(q[k] & 0xffff0000u), x[2 * k + 1], acc);
  }
  return acc;
}

// sum_e q_e * x_e over one 16-byte chunk of 32 int4 values (scale applied by the caller).
// Nibble p of 32-bit word k is element 8k + p. With the word xor 0x88888888 each nibble n is
// q + 8 in [0, 15]; 0x4B000000 | n is the float 2^23 + n exactly, so subtracting 2^23 + 8
// yields q exactly.
template <>
__device__ __forceinline__ float dot_chunk<WD_INT4>(const uint4& w, const float* x, float acc) {
  const uint32_t q[4] = {w.x ^ 0x88888888u, w.y ^ 0x88888888u, w.z ^ 0x88888888u, w.w ^ 0x88888888u};
#pragma unroll
  for (int k = 0; k < 4; k++) {
#pragma unroll
    for (int p = 0; p < 8; p++) {
      const float f = __uint_as_float(0x4B000000u | ((q[k] >> (4 * p)) & 0xFu)) - 8388616.0f;
      acc = fmaf(f, x[8 * k + p], acc);
    }
  }
  return acc;
}

// Lane-owned slice of an input vector: chunk c = j*32 + lane covers elements [c*EPC, (c+1)*EPC).
template <int WD, int CH>
__device__ __forceinline__ void load_vec(const void* x, int adtype, int n, int lane, float (&xr)[CH][Epc<WD>::v]) {
  constexpr int E = Epc<WD>::v;
#pragma unroll
  for (int j = 0; j < CH; j++) {
    const int base = (j * 32 + lane) * E;
#pragma unroll
    for (int e = 0; e < E; e++) {
      const int idx = base + e;
      float v = 0.f;
      if (idx < n) v = adtype ? bf16_bits(((const uint16_t*)x)[idx]) : ((const float*)x)[idx];
      xr[j][e] = v;
    }
  }
}

// ------------------------------------------------------------------------------------------
// Router: z_e = W_r[e] . h for every expert (one warp per row), then the last CTA to finish
// selects the top k (ties -> lower id), forms the gates and publishes them to host memory.

template <int WD, int CH>
__global__ void __launch_bounds__(256) k_router(const __grid_constant__ RouterArgs a) {
  constexpr int E = Epc<WD>::v;
  const int lane = threadIdx.x & 31;
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  const int64_t row_bytes = (int64_t)a.d * (WD == WD_FP32 ? 4 : 2);
  const int nch = (int)(row_bytes / 16);
  float xr[CH][E];
  load_vec<WD, CH>(a.h, a.adtype, a.d, lane, xr);
  for (int e = gw; e < a.E; e += nw) {
    const uint8_t* row = (const uint8_t*)a.w + (int64_t)e * row_bytes;
    uint4 w[CH];
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      w[j] = c < nch ? ld_stream(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
    }
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < CH; j++)
      if (j * 32 + lane < nch) acc = dot_chunk<WD>(w[j], xr[j], acc);
    acc = warp_sum(acc);
    if (lane == 0) a.z[e] = acc;
  }

  __shared__ int am_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned prev = atomicAdd(a.counter, 1u);
    am_last = (prev == gridDim.x - 1);
  }
  __syncthreads();
  if (!am_last || threadIdx.x >= 32) return;
  __threadfence();

  constexpr int PER = 8;  // E <= 256
  float v[PER];
  bool taken[PER];
#pragma unroll
  for (int j = 0; j < PER; j++) {
    const int e = j * 32 + lane;
    v[j] = e < a.E ? __ldcg(a.z + e) : -INFINITY;
    taken[j] = e >= a.E;
  }
  float my_z = -INFINITY;
  int my_i = -1;
  for (int r = 0; r < a.k; r++) {
    float bv = -INFINITY;
    int bi = 0x7fffffff;
#pragma unroll
    for (int j = 0; j < PER; j++) {
      const int e = j * 32 + lane;
      if (!taken[j] && (v[j] > bv || (v[j] == bv && e < bi))) {
        bv = v[j];
        bi = e;
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(kFull, bv, off);
      const int oi = __shfl_xor_sync(kFull, bi, off);
      if (ov > bv || (ov == bv && oi < bi)) {
        bv = ov;
        bi = oi;
      }
    }
    if (lane == r) {
      my_z = bv;
      my_i = bi;
    }
#pragma unroll
    for (int j = 0; j < PER; j++)
      if (bi == j * 32 + lane) taken[j] = true;
  }
  const float m = __shfl_sync(kFull, my_z, 0);
  const float ex = lane < a.k ? expf(my_z - m) : 0.f;
  float denom;
  if (a.renorm) {
    denom = warp_sum(ex);
  } else {
    float part = 0.f;
#pragma unroll
    for (int j = 0; j < PER; j++)
      if (j * 32 + lane < a.E) part += expf(v[j] - m);
    denom = warp_sum(part);
  }
  if (lane < a.k) {
    a.out->idx[lane] = my_i;
    a.out->gate[lane] = ex / denom;
  }
  __syncwarp();
  __threadfence_system();
  if (lane == 0) {
    *a.counter = 0u;
    a.out->seq = a.seq;
  }
}

// ------------------------------------------------------------------------------------------
// Gate-up: for every task t (an expert in a slot and an input x) and row i,
// u_t[i] = silu(W_g[i] . x) * (W_u[i] . x). One warp per (task, row pair); gate row i and up
// row i are adjacent in the slot image, so a warp streams 2 * row_bytes contiguous bytes.

template <int WD, int CH>
__global__ void __launch_bounds__(128) k_gateup(const __grid_constant__ GateUpArgs a) {
  constexpr int E = Epc<WD>::v;
  const int lane = threadIdx.x & 31;
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  const int64_t rb = a.lay.row_bytes_gu;
  const int nch = (int)(rb / 16);
  const int total = a.n_tasks * a.I;
  const int G = a.d / 128;
  float xr[CH][E];
  int cur = -1;
  for (int p = gw; p < total; p += nw) {
    const int t = p / a.I;
    const int i = p - t * a.I;
    if (t != cur) {
      load_vec<WD, CH>(a.t[t].x, a.adtype, a.d, lane, xr);
      cur = t;
    }
    const uint8_t* rg = a.t[t].blob + (int64_t)i * 2 * rb;
    const uint8_t* ru = rg + rb;
    uint4 wg[CH], wu[CH];
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      const bool ok = c < nch;
      wg[j] = ok ? ld_stream(rg + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
      wu[j] = ok ? ld_stream(ru + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
    }
    float ag = 0.f, au = 0.f;
    if (WD == WD_INT4) {
      const uint16_t* sc = (const uint16_t*)(a.t[t].blob + a.lay.gu_scale_off) + (int64_t)i * 2 * G;
#pragma unroll
      for (int j = 0; j < CH; j++) {
        const int c = j * 32 + lane;
        if (c < nch) {
          const int g = c >> 2;
          ag = fmaf(bf16_bits(sc[g]), dot_chunk<WD>(wg[j], xr[j], 0.f), ag);
          au = fmaf(bf16_bits(sc[G + g]), dot_chunk<WD>(wu[j], xr[j], 0.f), au);
        }
      }
    } else {
#pragma unroll
      for (int j = 0; j < CH; j++) {
        if (j * 32 + lane < nch) {
          ag = dot_chunk<WD>(wg[j], xr[j], ag);
          au = dot_chunk<WD>(wu[j], xr[j], au);
        }
      }
    }
    ag = warp_sum(ag);
    au = warp_sum(au);
    if (lane == 0) a.t[t].u[i] = ag / (1.0f + expf(-ag)) * au;
  }
}

// ------------------------------------------------------------------------------------------
// Down projection + combine: out[o] = sum_r g_r * (W_d^(r)[o] . u_r), ranks in order. All
// ranks' u vectors are staged in shared memory, padded by 4 floats per 32 so that the
// 16-byte reads of a warp spread over all banks. One warp per output row; the loads of four
// ranks are issued before their arithmetic.

__host__ __device__ __forceinline__ int upad(int i) { return i + 4 * (i >> 5); }

template <int WD, int CHD>
__global__ void __launch_bounds__(256) k_down_combine(const __grid_constant__ DownArgs a) {
  constexpr int E = Epc<WD>::v;
  extern __shared__ float4 smem4[];
  float* us = reinterpret_cast<float*>(smem4);
  const int ipad = upad(a.I + 31 - ((a.I + 31) & 31));
  for (int idx = threadIdx.x; idx < a.k * a.I; idx += blockDim.x) {
    const int r = idx / a.I;
    const int i = idx - r * a.I;
    us[r * ipad + upad(i)] = a.u[idx];
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  const int64_t rb = a.lay.row_bytes_d;
  const int nch = (int)(rb / 16);
  const int G = a.I / 128;
  for (int o = gw; o < a.d; o += nw) {
    float acc = 0.f;
    for (int r0 = 0; r0 < a.k; r0 += 4) {
      uint4 w[4][CHD];
#pragma unroll
      for (int rr = 0; rr < 4; rr++) {
        const int r = r0 + rr;
        const uint8_t* row = r < a.k ? a.blob[r] + a.lay.d_off + (int64_t)o * rb : nullptr;
#pragma unroll
        for (int j = 0; j < CHD; j++) {
          const int c = j * 32 + lane;
          w[rr][j] = (r < a.k && c < nch) ? ld_stream(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
        }
      }
#pragma unroll
      for (int rr = 0; rr < 4; rr++) {
        const int r = r0 + rr;
        if (r >= a.k) break;
        const float* ur = us + r * ipad;
        float part = 0.f;
#pragma unroll
        for (int j = 0; j < CHD; j++) {
          const int c = j * 32 + lane;
          if (c < nch) {
            float xv[E];
            const float4* src = reinterpret_cast<const float4*>(ur + upad(c * E));
#pragma unroll
            for (int q = 0; q < E / 4; q++) {
              const float4 f = src[q];
              xv[4 * q] = f.x;
              xv[4 * q + 1] = f.y;
              xv[4 * q + 2] = f.z;
              xv[4 * q + 3] = f.w;
            }
            if (WD == WD_INT4) {
              const uint16_t* sc = (const uint16_t*)(a.blob[r] + a.lay.d_scale_off) + (int64_t)o * G;
              part = fmaf(bf16_bits(sc[c >> 2]), dot_chunk<WD>(w[rr][j], xv, 0.f), part);
            } else {
              part = dot_chunk<WD>(w[rr][j], xv, part);
            }
          }
        }
        acc = fmaf(a.gate[r], part, acc);
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) {
      if (a.adtype)
        reinterpret_cast<__nv_bfloat16*>(a.out)[o] = __float2bfloat16_rn(acc);
      else
        reinterpret_cast<float*>(a.out)[o] = acc;
    }
  }
}

int g_num_sms = 0;

int num_sms() {
  if (g_num_sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_num_sms <= 0) g_num_sms = 1;
  }
  return g_num_sms;
}

int pick_ch(int nch) {
  const int need = (nch + 31) / 32;
  if (need <= 1) return 1;
  if (need <= 2) return 2;
  if (need <= 4) return 4;
  if (need <= 8) return 8;
  if (need <= 16) return 16;
  return -1;
}

int pick_chd(int nch) {
  const int need = (nch + 31) / 32;
  if (need <= 1) return 1;
  if (need <= 2) return 2;
  if (need <= 3) return 3;
  if (need <= 4) return 4;
  if (need <= 8) return 8;
  return -1;
}

template <int WD, int CH>
cudaError_t run_router(const RouterArgs& a, cudaStream_t s) {
  const int warps = 8;
  const int grid = (a.E + warps - 1) / warps;
  k_router<WD, CH><<<grid, warps * 32, 0, s>>>(a);
  return cudaGetLastError();
}

template <int WD, int CH>
cudaError_t run_gateup(const GateUpArgs& a, cudaStream_t s) {
  const int total = a.n_tasks * a.I;
  if (total <= 0) return cudaSuccess;
  static int occ = 0;
  if (occ == 0) {
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_gateup<WD, CH>, 128, 0);
    if (occ < 1) occ = 1;
  }
  int grid = (total + 3) / 4;
  const int cap = num_sms() * occ;
  if (grid > cap) grid = cap;
  k_gateup<WD, CH><<<grid, 128, 0, s>>>(a);
  return cudaGetLastError();
}

template <int WD, int CHD>
cudaError_t run_down(const DownArgs& a, cudaStream_t s) {
  const int ipad = upad(a.I + 31 - ((a.I + 31) & 31));
  const size_t smem = (size_t)a.k * ipad * sizeof(float);
  static size_t smem_set = 48 * 1024;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(k_down_combine<WD, CHD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  static size_t occ_smem = (size_t)-1;
  static int occ = 0;
  if (occ_smem != smem) {
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_down_combine<WD, CHD>, 256, smem);
    if (occ < 1) occ = 1;
    occ_smem = smem;
  }
  int grid = (a.d + 7) / 8;
  const int cap = num_sms() * occ;
  if (grid > cap) grid = cap;
  k_down_combine<WD, CHD><<<grid, 256, smem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_router(const RouterArgs& a, cudaStream_t s) {
  const int64_t rb = (int64_t)a.d * (a.wdtype == WD_FP32 ? 4 : 2);
  const int ch = pick_ch((int)(rb / 16));
#define MOE_R(WD)                                         \
  switch (ch) {                                           \
    case 1: return run_router<WD, 1>(a, s);               \
    case 2: return run_router<WD, 2>(a, s);               \
    case 4: return run_router<WD, 4>(a, s);               \
    case 8: return run_router<WD, 8>(a, s);               \
    case 16: return run_router<WD, 16>(a, s);             \
    default: return cudaErrorInvalidValue;                \
  }
  if (a.wdtype == WD_FP32) {
    MOE_R(WD_FP32)
  } else {
    MOE_R(WD_BF16)
  }
#undef MOE_R
}

cudaError_t launch_gateup(const GateUpArgs& a, int wdtype, cudaStream_t s) {
  const int ch = pick_ch((int)(a.lay.row_bytes_gu / 16));
#define MOE_G(WD)                                         \
  switch (ch) {                                           \
    case 1: return run_gateup<WD, 1>(a, s);               \
    case 2: return run_gateup<WD, 2>(a, s);               \
    case 4: return run_gateup<WD, 4>(a, s);               \
    case 8: return run_gateup<WD, 8>(a, s);               \
    case 16: return run_gateup<WD, 16>(a, s);             \
    default: return cudaErrorInvalidValue;                \
  }
  if (wdtype == WD_FP32) {
    MOE_G(WD_FP32)
  } else if (wdtype == WD_BF16) {
    MOE_G(WD_BF16)
  } else {
    MOE_G(WD_INT4)
  }
#undef MOE_G
}

cudaError_t launch_down_combine(const DownArgs& a, int wdtype, cudaStream_t s) {
  const int ch = pick_chd((int)(a.lay.row_bytes_d / 16));
#define MOE_D(WD)                                         \
  switch (ch) {                                           \
    case 1: return run_down<WD, 1>(a, s);                 \
    case 2: return run_down<WD, 2>(a, s);                 \
    case 3: return run_down<WD, 3>(a, s);                 \
    case 4: return run_down<WD, 4>(a, s);                 \
    case 8: return run_down<WD, 8>(a, s);                 \
    default: return cudaErrorInvalidValue;                \
  }
  if (wdtype == WD_FP32) {
    MOE_D(WD_FP32)
  } else if (wdtype == WD_BF16) {
    MOE_D(WD_BF16)
  } else {
    MOE_D(WD_INT4)
  }
#undef MOE_D
}

}  // namespace moe
