// Router / top-k, SwiGLU gate-up GEMV and down-projection + combine kernels (sm_103a).
//
// At batch 1 every kernel streams weights from HBM once, so each is written for latency as
// much as bandwidth: a warp issues all 128-bit streaming loads (L1 no-allocate) of its rows
// before it waits on anything, the activation vector is staged in shared memory with 16-byte
// loads while those weight loads are in flight, row dot products are reduced with a fixed
// XOR-shuffle butterfly, and accumulation is fp32. No reduction order depends on which slot an
// expert occupies or on the grid size, so results are bit-identical between capped and
// uncapped pools.
#include <cooperative_groups.h>

#include <algorithm>
#include <cuda_bf16.h>
#include <math.h>

#include "dev.cuh"
#include "kernels.cuh"

namespace cg = cooperative_groups;

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

using namespace dev;

// ------------------------------------------------------------------------------------------
// Router. One thread-block cluster of 8 CTAs x 16 warps: warp w of the cluster computes the
// logits z_e = W_r[e] . h of rows e = w, w + 128, ... and stores them into CTA 0's shared
// memory (distributed shared memory); after a cluster barrier one warp of CTA 0 selects the
// top k (ties -> lower id), forms the gates and publishes them to host-mapped memory.

constexpr int kRouterCtas = 8;
constexpr int kRouterWarps = 16;

template <int WD, int CH>
__global__ void __launch_bounds__(kRouterWarps * 32) k_router(const __grid_constant__ RouterArgs a) {
  extern __shared__ uint4 xs4[];
  __shared__ float zs[256];
  const uint8_t* xs = reinterpret_cast<const uint8_t*>(xs4);
  cg::cluster_group cluster = cg::this_cluster();
  const unsigned crank = cluster.block_rank();
  const int lane = threadIdx.x & 31;
  const int gw = (int)crank * kRouterWarps + (threadIdx.x >> 5);
  constexpr int kW = kRouterCtas * kRouterWarps;
  const int64_t rb = (int64_t)a.d * (WD == WD_FP32 ? 4 : 2);
  const int nch = (int)(rb / 16);
  float* zl = cluster.map_shared_rank(zs, 0);

  // every CTA of the cluster must be running before its shared memory is written remotely
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  uint4 w[CH];
  const bool ok0 = gw < a.E;
  {
    const uint8_t* row = (const uint8_t*)a.w + (int64_t)(ok0 ? gw : 0) * rb;
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      w[j] = (ok0 && c < nch) ? ld_stream(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
    }
  }
  stage16(xs4, a.h, a.d * (WD == WD_FP32 ? 4 : 2), threadIdx.x, blockDim.x);
  __syncthreads();
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
  for (int e = gw; e < a.E; e += kW) {
    if (e != gw) {
      const uint8_t* row = (const uint8_t*)a.w + (int64_t)e * rb;
#pragma unroll
      for (int j = 0; j < CH; j++) {
        const int c = j * 32 + lane;
        w[j] = c < nch ? ld_stream(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
      }
    }
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      if (c < nch) acc = dot_chunk<WD>(w[j], xs + (int64_t)c * Tr<WD>::xbytes, acc);
    }
    acc = warp_sum(acc);
    if (lane == 0) zl[e] = acc;
  }
  cluster.sync();
  if (crank != 0 || threadIdx.x >= 32) return;

  constexpr int PER = 8;  // E <= 256
  uint32_t key[PER];
#pragma unroll
  for (int j = 0; j < PER; j++) {
    const int e = j * 32 + lane;
    key[j] = e < a.E ? ord_key(zs[e]) : 0u;  // 0: below every real key, never selected
  }
  float my_z = 0.f;
  int my_i = -1;
  for (int r = 0; r < a.k; r++) {
    uint32_t bk = 0u;
    int bi = 0x7fffffff;
#pragma unroll
    for (int j = 0; j < PER; j++) {
      if (key[j] > bk) {  // ascending j: an equal key later never replaces (lower id wins)
        bk = key[j];
        bi = j * 32 + lane;
      }
    }
    const uint32_t mk = __reduce_max_sync(kFull, bk);
    const int win = (int)__reduce_min_sync(kFull, bk == mk ? (uint32_t)bi : 0xffffffffu);
    if (lane == r) {
      my_z = key_value(mk);
      my_i = win;
    }
#pragma unroll
    for (int j = 0; j < PER; j++)
      if (win == j * 32 + lane) key[j] = 0u;
  }
  const float m = __shfl_sync(kFull, my_z, 0);
  const float ex = lane < a.k ? expf(my_z - m) : 0.f;
  float denom;
  if (a.renorm) {
    denom = warp_sum(ex);
  } else {
    float part = 0.f;
    for (int e = lane; e < a.E; e += 32) part += expf(zs[e] - m);
    denom = warp_sum(part);
  }
  if (lane < a.k) {
    a.out->idx[lane] = my_i;
    a.out->gate[lane] = ex / denom;
  }
  if (a.want_z)
    for (int e = lane; e < a.E; e += 32) a.out->z[e] = zs[e];
  __syncwarp();
  __threadfence_system();
  if (lane == 0) a.out->seq = a.seq;
}

// ------------------------------------------------------------------------------------------
// Gate-up: u_t[i] = silu(W_g[i] . x) * (W_u[i] . x). One warp per (task, row pair); gate row i
// and up row i are adjacent in the slot image, so a warp streams 2 * row_bytes contiguous
// bytes. Weight loads are issued before the CTA stages x.

constexpr int kGuWarps = 4;

template <int WD, int CH>
__global__ void __launch_bounds__(kGuWarps * 32) k_gateup(const __grid_constant__ GateUpArgs a) {
  extern __shared__ uint4 xs4[];
  const uint8_t* xs = reinterpret_cast<const uint8_t*>(xs4);
  const int lane = threadIdx.x & 31;
  const int p = blockIdx.x * kGuWarps + (threadIdx.x >> 5);
  const int64_t rb = a.lay.row_bytes_gu;
  const int nch = (int)(rb / 16);
  const bool valid = p < a.n_tasks * a.I;
  const int t = valid ? p / a.I : 0;
  const int i = valid ? p - t * a.I : 0;
  const uint8_t* rg = a.blob[t] + (int64_t)i * 2 * rb;
  const uint8_t* ru = rg + rb;
  uint4 wg[CH], wu[CH];
#pragma unroll
  for (int j = 0; j < CH; j++) {
    const int c = j * 32 + lane;
    const bool ok = valid && c < nch;
    wg[j] = ok ? ld_stream(rg + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
    wu[j] = ok ? ld_stream(ru + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
  }
  float sg[CH], su[CH];
  if (WD == WD_INT4) {
    const int G = a.d / 128;
    const uint16_t* sc = (const uint16_t*)(a.blob[t] + a.lay.gu_scale_off) + (int64_t)i * 2 * G;
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      const bool ok = valid && c < nch;
      sg[j] = ok ? bf16_bits(__ldg(sc + (c >> 2))) : 0.f;
      su[j] = ok ? bf16_bits(__ldg(sc + G + (c >> 2))) : 0.f;
    }
  }
  stage16(xs4, a.x, a.d * (WD == WD_FP32 ? 4 : 2), threadIdx.x, blockDim.x);
  __syncthreads();
  if (!valid) return;
  float ag = 0.f, au = 0.f;
#pragma unroll
  for (int j = 0; j < CH; j++) {
    const int c = j * 32 + lane;
    if (c < nch) {
      const uint8_t* xc = xs + (int64_t)c * Tr<WD>::xbytes;
      if (WD == WD_INT4) {
        ag = fmaf(sg[j], dot_chunk<WD>(wg[j], xc, 0.f), ag);
        au = fmaf(su[j], dot_chunk<WD>(wu[j], xc, 0.f), au);
      } else {
        ag = dot_chunk<WD>(wg[j], xc, ag);
        au = dot_chunk<WD>(wu[j], xc, au);
      }
    }
  }
  ag = warp_sum(ag);
  au = warp_sum(au);
  if (lane == 0) a.u[t][i] = ag / (1.0f + expf(-ag)) * au;
}

// ------------------------------------------------------------------------------------------
// Down projection + combine: out[o] = sum_r g_r * (W_d^(r)[o] . u_r), ranks in order. One warp
// per output row issues the loads of up to 8 ranks' rows at once, then the CTA stages all u
// vectors in shared memory (padded by 4 floats per 32 so 16-byte reads spread over all banks).

constexpr int kDnWarps = 8;
// ranks whose rows are in flight together: about 24 chunks (384 B) per lane
template <int CHD>
struct DnRanks {
  static constexpr int v = 24 / CHD > 8 ? 8 : 24 / CHD;
};

template <int WD, int CHD>
__global__ void __launch_bounds__(kDnWarps * 32) k_down_combine(const __grid_constant__ DownArgs a) {
  constexpr int E = Tr<WD>::epc;
  constexpr int kDnRanks = DnRanks<CHD>::v;
  extern __shared__ float4 us4[];
  float* us = reinterpret_cast<float*>(us4);
  const int lane = threadIdx.x & 31;
  const int o = blockIdx.x * kDnWarps + (threadIdx.x >> 5);
  const bool valid = o < a.d;
  const int64_t rb = a.lay.row_bytes_d;
  const int nch = (int)(rb / 16);
  const int G = a.I / 128;
  const int ipad = ipad_of(a.I);

  uint4 w[kDnRanks][CHD];
  float sc[kDnRanks][CHD];
  auto issue = [&](int r0) {
#pragma unroll
    for (int rr = 0; rr < kDnRanks; rr++) {
      const int r = r0 + rr;
      const bool rok = valid && r < a.k;
      const uint8_t* row = a.blob[rok ? r : 0] + a.lay.d_off + (int64_t)(valid ? o : 0) * rb;
#pragma unroll
      for (int j = 0; j < CHD; j++) {
        const int c = j * 32 + lane;
        w[rr][j] = (rok && c < nch) ? ld_stream(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
        if (WD == WD_INT4) {
          const uint16_t* s = (const uint16_t*)(a.blob[rok ? r : 0] + a.lay.d_scale_off) + (int64_t)(valid ? o : 0) * G;
          sc[rr][j] = (rok && c < nch) ? bf16_bits(__ldg(s + (c >> 2))) : 0.f;
        }
      }
    }
  };
  issue(0);
  // stage u: float4 q holds elements 4q..4q+3 of the rank-major [k x I] array (I % 4 == 0)
  {
    const float4* u4 = reinterpret_cast<const float4*>(a.u);
    const int n4 = a.k * a.I / 4;
#pragma unroll 4
    for (int q = threadIdx.x; q < n4; q += blockDim.x) {
      const float4 v = __ldg(u4 + q);
      const int r = (4 * q) / a.I;
      const int i = 4 * q - r * a.I;
      *reinterpret_cast<float4*>(us + r * ipad + upad(i)) = v;
    }
  }
  __syncthreads();
  if (!valid) return;
  float acc = 0.f;
  for (int r0 = 0; r0 < a.k; r0 += kDnRanks) {
    if (r0 > 0) issue(r0);
#pragma unroll
    for (int rr = 0; rr < kDnRanks; rr++) {
      const int r = r0 + rr;
      if (r >= a.k) break;
      const float* ur = us + r * ipad;
      float part = 0.f;
#pragma unroll
      for (int j = 0; j < CHD; j++) {
        const int c = j * 32 + lane;
        if (c < nch) {
          if (WD == WD_INT4)
            part = fmaf(sc[rr][j], dot_chunk_u<WD>(w[rr][j], ur + upad(c * E), 0.f), part);
          else
            part = dot_chunk_u<WD>(w[rr][j], ur + upad(c * E), part);
        }
      }
      acc = fmaf(a.gate[r], part, acc);
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) {
    if (WD == WD_FP32)
      reinterpret_cast<float*>(a.out)[o] = acc;
    else
      reinterpret_cast<__nv_bfloat16*>(a.out)[o] = __float2bfloat16_rn(acc);
  }
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
  if (need <= 6) return 6;
  if (need <= 8) return 8;
  return -1;
}

// Opt the kernel in to `smem` bytes of dynamic shared memory on the current device when that is
// above the default 48 KB (the attribute is per device, so it is set at every such launch).
template <typename K>
cudaError_t allow_smem(K kernel, size_t smem) {
  if (smem <= 48 * 1024) return cudaSuccess;
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

template <int WD, int CH>
cudaError_t run_router(const RouterArgs& a, cudaStream_t s) {
  const size_t smem = (size_t)a.d * (WD == WD_FP32 ? 4 : 2);
  cudaError_t e = allow_smem(k_router<WD, CH>, smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kRouterCtas);
  cfg.blockDim = dim3(kRouterWarps * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kRouterCtas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_router<WD, CH>, a);
}

template <int WD, int CH>
cudaError_t run_gateup(const GateUpArgs& a, cudaStream_t s) {
  const int total = a.n_tasks * a.I;
  if (total <= 0) return cudaSuccess;
  const size_t smem = (size_t)a.d * (WD == WD_FP32 ? 4 : 2);
  cudaError_t e = allow_smem(k_gateup<WD, CH>, smem);
  if (e != cudaSuccess) return e;
  k_gateup<WD, CH><<<(total + kGuWarps - 1) / kGuWarps, kGuWarps * 32, smem, s>>>(a);
  return cudaGetLastError();
}

template <int WD, int CHD>
cudaError_t run_down(const DownArgs& a, cudaStream_t s) {
  const size_t smem = (size_t)a.k * ipad_of(a.I) * sizeof(float);
  cudaError_t e = allow_smem(k_down_combine<WD, CHD>, smem);
  if (e != cudaSuccess) return e;
  k_down_combine<WD, CHD><<<(a.d + kDnWarps - 1) / kDnWarps, kDnWarps * 32, smem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_router(const RouterArgs& a, cudaStream_t s) {
  const int64_t rb = (int64_t)a.d * (a.wdtype == WD_FP32 ? 4 : 2);
  const int ch = pick_ch((int)(rb / 16));
#define MOE_R(WD)                             \
  switch (ch) {                               \
    case 1: return run_router<WD, 1>(a, s);   \
    case 2: return run_router<WD, 2>(a, s);   \
    case 4: return run_router<WD, 4>(a, s);   \
    case 8: return run_router<WD, 8>(a, s);   \
    case 16: return run_router<WD, 16>(a, s); \
    default: return cudaErrorInvalidValue;    \
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
#define MOE_G(WD)                             \
  switch (ch) {                               \
    case 1: return run_gateup<WD, 1>(a, s);   \
    case 2: return run_gateup<WD, 2>(a, s);   \
    case 4: return run_gateup<WD, 4>(a, s);   \
    case 8: return run_gateup<WD, 8>(a, s);   \
    case 16: return run_gateup<WD, 16>(a, s); \
    default: return cudaErrorInvalidValue;    \
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

namespace {

__global__ void __launch_bounds__(256) k_touch_pages(const uint8_t* base, int64_t bytes, int shift) {
  const int64_t pages = (bytes + (1ll << shift) - 1) >> shift;
  for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < pages; p += (int64_t)gridDim.x * blockDim.x)
    asm volatile("{ .reg .u32 t; ld.volatile.global.u32 t, [%0]; }" ::"l"(base + (p << shift)) : "memory");
}

}  // namespace

cudaError_t launch_touch_pages(const uint8_t* base, int64_t bytes, int shift, cudaStream_t s) {
  if (bytes <= 0) return cudaSuccess;
  const int64_t pages = (bytes + (1ll << shift) - 1) >> shift;
  const int blocks = (int)std::min<int64_t>((pages + 255) / 256, 1024);
  k_touch_pages<<<blocks, 256, 0, s>>>(base, bytes, shift);
  return cudaGetLastError();
}

cudaError_t launch_down_combine(const DownArgs& a, int wdtype, cudaStream_t s) {
  const int ch = pick_chd((int)(a.lay.row_bytes_d / 16));
#define MOE_D(WD)                           \
  switch (ch) {                             \
    case 1: return run_down<WD, 1>(a, s);   \
    case 2: return run_down<WD, 2>(a, s);   \
    case 3: return run_down<WD, 3>(a, s);   \
    case 4: return run_down<WD, 4>(a, s);   \
    case 6: return run_down<WD, 6>(a, s);   \
    case 8: return run_down<WD, 8>(a, s);   \
    default: return cudaErrorInvalidValue;  \
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
