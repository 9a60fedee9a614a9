// Chained decoder blocks around the MoE layer: one decode token at batch 1 through a stack whose
// layers feed one another, the paper's end-to-end setting (a whole MoE decoder at a 4096-token
// context, Sec. "Experimental Setup"). The paper prints no architecture; the block is a
// Qwen3-MoE-class reading. Per layer l, with the fp32 residual stream x at position p:
//   a = RMSNorm(x) * w_in;  [q; k; v] = [W_q; W_k; W_v] a
//   q_h = RoPE(RMSNorm(q_h) * w_q, p),  k_g = RoPE(RMSNorm(k_g) * w_k, p);  (k_g, v_g) -> cache row p
//   o = grouped-query attention of q over cache rows 0..p;  x += W_o o
//   m = RMSNorm(x) * w_post;  x += MoE_l(m)
// MoE_l is layer l of the handle's fused decode kernel (routing, residency step of the shared slot
// group, expert FFN, combine), launched on its own: layer l + 1 routes on what layer l produced,
// so the residency sees real cross-layer dependence and no layer can be routed ahead.
//
// Precision: weights, caches and the MoE's input/output in the handle's activation storage (fp32,
// or bf16 for bf16 and int4 experts); the residual stream, norms, projections, rotary rotation
// and attention in fp32, with the rotary angle formed in fp64.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "moe.h"
#include "moe_internal.h"

namespace {

constexpr int kNormThreads = 1024;
constexpr int kGemvWarps = 8;
constexpr int kMaxGemvCols = 12288;  // activation staged in 48 KiB of shared memory

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) {
  return v;
}
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

// Sum over the CTA (blockDim.x a multiple of 32); every thread receives the total.
__device__ float block_sum(float v) {
  __shared__ float red[32];
  __shared__ float total;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[w] = v;
  __syncthreads();
  if (w == 0) {
    float t = lane < (int)(blockDim.x >> 5) ? red[lane] : 0.f;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
    if (lane == 0) total = t;
  }
  __syncthreads();
  return total;
}

// Residual stream entering layer l: x = x_in (layer 0, activation storage) or x + prev (the
// previous layer's MoE output); then a = RMSNorm(x) * w. One CTA. Optional logs: x, and prev
// as read.
template <typename T>
__global__ void __launch_bounds__(kNormThreads) k_dec_input(const T* x_in, const T* prev, float* x, const T* w,
                                                            int d, float eps, float* a, float* log_x,
                                                            float* log_prev) {
  float ss = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    float v;
    if (x_in) {
      v = to_f(x_in[i]);
    } else {
      const float p = to_f(prev[i]);
      v = x[i] + p;
      if (log_prev) log_prev[i] = p;
    }
    x[i] = v;
    if (log_x) log_x[i] = v;
    ss = fmaf(v, v, ss);
  }
  const float r = 1.0f / sqrtf(block_sum(ss) / (float)d + eps);
  for (int i = threadIdx.x; i < d; i += blockDim.x) a[i] = to_f(w[i]) * (x[i] * r);
}

// The MoE layer's input: m = RMSNorm(x) * w, stored in the activation storage. One CTA.
template <typename T>
__global__ void __launch_bounds__(kNormThreads) k_dec_post_norm(const float* x, const T* w, int d, float eps, T* m,
                                                                float* log_m) {
  float ss = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) ss = fmaf(x[i], x[i], ss);
  const float r = 1.0f / sqrtf(block_sum(ss) / (float)d + eps);
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const T q = from_f<T>(to_f(w[i]) * (x[i] * r));
    m[i] = q;
    if (log_m) log_m[i] = to_f(q);
  }
}

// After the last layer: x += prev (its MoE output); x_out = x.
template <typename T>
__global__ void k_dec_output(float* x, const T* prev, int d, float* x_out, float* log_prev) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < d; i += gridDim.x * blockDim.x) {
    const float p = to_f(prev[i]);
    const float v = x[i] + p;
    x[i] = v;
    x_out[i] = v;
    if (log_prev) log_prev[i] = p;
  }
}

// Dot product of one 16-byte chunk of a weight row with the matching activations.
__device__ __forceinline__ float dot16(const uint4 w, const float* act, float s) {
  const float4 a0 = *reinterpret_cast<const float4*>(act);
  s = fmaf(__uint_as_float(w.x), a0.x, s);
  s = fmaf(__uint_as_float(w.y), a0.y, s);
  s = fmaf(__uint_as_float(w.z), a0.z, s);
  return fmaf(__uint_as_float(w.w), a0.w, s);
}
__device__ __forceinline__ float dot16_bf16(const uint4 w, const float* act, float s) {
  const float4 a0 = *reinterpret_cast<const float4*>(act);
  const float4 a1 = *reinterpret_cast<const float4*>(act + 4);
  s = fmaf(__uint_as_float(w.x << 16), a0.x, s);
  s = fmaf(__uint_as_float(w.x & 0xffff0000u), a0.y, s);
  s = fmaf(__uint_as_float(w.y << 16), a0.z, s);
  s = fmaf(__uint_as_float(w.y & 0xffff0000u), a0.w, s);
  s = fmaf(__uint_as_float(w.z << 16), a1.x, s);
  s = fmaf(__uint_as_float(w.z & 0xffff0000u), a1.y, s);
  s = fmaf(__uint_as_float(w.w << 16), a1.z, s);
  return fmaf(__uint_as_float(w.w & 0xffff0000u), a1.w, s);
}

// y_r = W_r . act for the rows of W [rows x cols] (row-major, every row 16-byte aligned), with the
// fp32 activation staged in shared memory; one warp per row, 16-byte coalesced loads. acc != NULL
// adds y_r into acc[r] (one writer per row); y and log, where given, receive y_r.
template <typename T>
__global__ void __launch_bounds__(kGemvWarps * 32) k_dec_gemv(const T* W, int rows, int cols, const float* act,
                                                              float* y, float* acc, float* log) {
  extern __shared__ float4 s_act4[];
  float* s_act = reinterpret_cast<float*>(s_act4);
  for (int i = threadIdx.x; i < cols; i += blockDim.x) s_act[i] = act[i];
  __syncthreads();
  constexpr int EPC = 16 / (int)sizeof(T);  // elements per 16-byte chunk
  const int lane = threadIdx.x & 31;
  const int nch = cols / EPC;
  constexpr int U = 8;  // chunks in flight per lane: the loads of a batch are issued before any is used
  for (int r = blockIdx.x * kGemvWarps + (threadIdx.x >> 5); r < rows; r += gridDim.x * kGemvWarps) {
    const uint4* row = reinterpret_cast<const uint4*>(W + (int64_t)r * cols);
    float s = 0.f;
    for (int c0 = lane; c0 < nch; c0 += 32 * U) {
      uint4 w[U];
#pragma unroll
      for (int j = 0; j < U; j++) {
        const int c = c0 + 32 * j;
        w[j] = c < nch ? __ldg(row + c) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int j = 0; j < U; j++) {
        const int c = c0 + 32 * j;
        if (c < nch) {  // chunks in ascending order per lane, as one at a time would take them
          if constexpr (sizeof(T) == 4)
            s = dot16(w[j], s_act + c * EPC, s);
          else
            s = dot16_bf16(w[j], s_act + c * EPC, s);
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) {
      if (acc) acc[r] += s;
      if (y) y[r] = s;
      if (log) log[r] = s;
    }
  }
}

// One CTA per head, D threads (D = 64 or 128): query heads [0, Hq), key heads [Hq, Hq + Hkv) and
// value heads [Hq + Hkv, Hq + 2 Hkv) of qkv. A query or key head is normalised (RMSNorm over D
// with w_q or w_k) and rotated for position pos: element i pairs with i + D/2 (rotate-half), by
// the angle pos * theta^(-2i/D), formed in fp64 so that positions in the thousands keep fp32
// accuracy. Query heads go to q (fp32), key heads to cache row pos of Kc, value heads (as
// projected) to row pos of Vc.
template <typename T>
__global__ void __launch_bounds__(128) k_dec_heads(const float* qkv, int Hq, int Hkv, const T* wq, const T* wk,
                                                   float eps, int64_t pos, double theta, float* q, T* Kc, T* Vc,
                                                   int64_t max_pos) {
  __shared__ float s_n[128];
  const int D = blockDim.x;
  const int h = blockIdx.x, t = threadIdx.x;
  const float v = qkv[(int64_t)h * D + t];
  if (h >= Hq + Hkv) {
    Vc[((int64_t)(h - Hq - Hkv) * max_pos + pos) * D + t] = from_f<T>(v);
    return;
  }
  const bool is_q = h < Hq;
  const float r = 1.0f / sqrtf(block_sum(v * v) / (float)D + eps);
  const float n = to_f(is_q ? wq[t] : wk[t]) * (v * r);
  s_n[t] = n;
  __syncthreads();
  const int half = D / 2;
  const int i = t < half ? t : t - half;
  double sn, cs;
  sincos((double)pos * pow(theta, -2.0 * (double)i / (double)D), &sn, &cs);
  const float c = (float)cs, s = (float)sn;
  const float out = t < half ? n * c - s_n[t + half] * s : n * c + s_n[t - half] * s;
  if (is_q)
    q[(int64_t)h * D + t] = out;
  else
    Kc[((int64_t)(h - Hq) * max_pos + pos) * D + t] = from_f<T>(out);
}

struct DecLayer {
  uint8_t* mem = nullptr;  // one allocation: wqkv, wo, norms, K cache, V cache
  void* wqkv = nullptr;    // [(Hq + 2 Hkv) D x d]: W_q rows, then W_k, then W_v
  void* wo = nullptr;      // [d x Hq D]
  void* norms = nullptr;   // w_in [d], w_post [d], w_q [D], w_k [D]
  void* K = nullptr;       // [Hkv x max_pos x D]
  void* V = nullptr;
  bool set = false;
  int64_t n_pos = 0;       // cache rows written
};

size_t align256(size_t n) { return (n + 255) & ~(size_t)255; }

}  // namespace

struct moe_decoder {
  moe_handle* moe = nullptr;
  moe::MoeShape shape{};
  moe_decoder_config cfg{};
  int64_t es = 0;  // element bytes of the weights, caches and MoE activations
  int qrows = 0, kvrows = 0;
  size_t off_wo = 0, off_norms = 0, off_k = 0, off_v = 0, layer_bytes = 0;
  std::vector<DecLayer> layers;
  uint8_t* work = nullptr;  // x, a, qkv, q, o (fp32), attention partials, MoE input / output rows
  float* x = nullptr;
  float* a = nullptr;
  float* qkv = nullptr;
  float* q = nullptr;
  float* o = nullptr;
  float* part = nullptr;
  void* hid = nullptr;   // [L x d] activation storage: the MoE layers' inputs
  void* mout = nullptr;  // [L x d]: their outputs
  std::string err;
};

namespace {

thread_local std::string g_create_err;

moe_status dfail(moe_decoder* dec, moe_status st, const std::string& msg) {
  if (dec)
    dec->err = msg;
  else
    g_create_err = msg;
  return st;
}

void free_decoder(moe_decoder* dec) {
  for (DecLayer& ly : dec->layers) cudaFree(ly.mem);
  cudaFree(dec->work);
  cudaGetLastError();
}

template <typename T>
moe_status run_step(moe_decoder* dec, const void* x_in, float* x_out, float* log, cudaStream_t s) {
  const moe::MoeShape& sh = dec->shape;
  const moe_decoder_config& c = dec->cfg;
  const int L = sh.n_layers, d = sh.d, D = c.head_dim;
  const int64_t pos = dec->layers[0].n_pos;
  const float eps = (float)c.eps;
  const int qkv_rows = dec->qrows + 2 * dec->kvrows;
  T* hid = (T*)dec->hid;
  T* mout = (T*)dec->mout;
  auto launched = [&](const char* what) -> moe_status {
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? MOE_OK : dfail(dec, MOE_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
  };
  moe_status st;
  for (int l = 0; l < L; l++) {
    const DecLayer& ly = dec->layers[l];
    const T* norms = (const T*)ly.norms;
    float* lg = log ? log + (int64_t)l * 4 * d : nullptr;
    k_dec_input<T><<<1, kNormThreads, 0, s>>>(l == 0 ? (const T*)x_in : nullptr,
                                              l == 0 ? nullptr : mout + (int64_t)(l - 1) * d, dec->x, norms, d, eps,
                                              dec->a, lg, (log && l > 0) ? log + ((int64_t)(l - 1) * 4 + 3) * d : nullptr);
    if ((st = launched("input norm")) != MOE_OK) return st;
    k_dec_gemv<T><<<(qkv_rows + kGemvWarps - 1) / kGemvWarps, kGemvWarps * 32, d * sizeof(float), s>>>(
        (const T*)ly.wqkv, qkv_rows, d, dec->a, dec->qkv, nullptr, nullptr);
    if ((st = launched("q/k/v projection")) != MOE_OK) return st;
    k_dec_heads<T><<<c.n_heads + 2 * c.n_kv_heads, D, 0, s>>>(dec->qkv, c.n_heads, c.n_kv_heads, norms + 2 * d,
                                                              norms + 2 * d + D, eps, pos, c.rope_theta, dec->q,
                                                              (T*)ly.K, (T*)ly.V, c.max_pos);
    if ((st = launched("head norms and rotary")) != MOE_OK) return st;
    cudaError_t e = moe::attention_launch(sh.adtype, dec->q, ly.K, ly.V, c.n_heads, c.n_kv_heads, D, c.max_pos,
                                          pos + 1, dec->o, dec->part, s);
    if (e != cudaSuccess) return dfail(dec, MOE_ERR_CUDA, std::string("attention: ") + cudaGetErrorString(e));
    k_dec_gemv<T><<<(d + kGemvWarps - 1) / kGemvWarps, kGemvWarps * 32, dec->qrows * sizeof(float), s>>>(
        (const T*)ly.wo, d, dec->qrows, dec->o, nullptr, dec->x, lg ? lg + d : nullptr);
    if ((st = launched("output projection")) != MOE_OK) return st;
    k_dec_post_norm<T><<<1, kNormThreads, 0, s>>>(dec->x, norms + d, d, eps, hid + (int64_t)l * d,
                                                  lg ? lg + 2 * d : nullptr);
    if ((st = launched("post-attention norm")) != MOE_OK) return st;
    st = moe::moe_run_layer(dec->moe, dec->hid, dec->mout, l, s);
    if (st != MOE_OK) return dfail(dec, st, std::string("MoE layer: ") + moe::moe_error_text(dec->moe));
  }
  k_dec_output<T><<<(d + 255) / 256, 256, 0, s>>>(dec->x, mout + (int64_t)(L - 1) * d, d, x_out,
                                                  log ? log + ((int64_t)(L - 1) * 4 + 3) * d : nullptr);
  return launched("output");
}

}  // namespace

extern "C" {

moe_status moe_decoder_create(moe_handle* moe, const moe_decoder_config* cfg, moe_decoder** out) {
  if (!out) return dfail(nullptr, MOE_ERR_INVALID, "out is NULL");
  *out = nullptr;
  if (!moe || !cfg) return dfail(nullptr, MOE_ERR_INVALID, "NULL handle or config");
  moe::MoeShape sh{};
  moe::moe_shape(moe, &sh);
  if (!sh.device_batch1)
    return dfail(nullptr, MOE_ERR_INVALID, "the MoE handle must use the device schedule with max_batch 1");
  const moe_decoder_config& c = *cfg;
  if (!moe::attention_shape_ok(c.n_heads, c.n_kv_heads, c.head_dim))
    return dfail(nullptr, MOE_ERR_INVALID, "head_dim must be 64 or 128 and n_heads / n_kv_heads 1, 2, 4 or 8");
  if (c.max_pos < 1) return dfail(nullptr, MOE_ERR_INVALID, "max_pos must be positive");
  if (!(c.eps > 0.0) || !(c.rope_theta > 0.0)) return dfail(nullptr, MOE_ERR_INVALID, "eps and rope_theta must be positive");
  const int64_t es = sh.adtype == MOE_DTYPE_FP32 ? 4 : 2;
  const int64_t qrows = (int64_t)c.n_heads * c.head_dim, kvrows = (int64_t)c.n_kv_heads * c.head_dim;
  if ((sh.d * es) % 16 || sh.d > kMaxGemvCols || qrows > kMaxGemvCols)
    return dfail(nullptr, MOE_ERR_INVALID, "d must be a multiple of 16 bytes of activations, d and n_heads * head_dim at most 12288");
  moe_decoder* dec = new moe_decoder();
  dec->moe = moe;
  dec->shape = sh;
  dec->cfg = c;
  dec->es = es;
  dec->qrows = (int)qrows;
  dec->kvrows = (int)kvrows;
  const size_t wqkv = (size_t)(qrows + 2 * kvrows) * sh.d * es, wo = (size_t)sh.d * qrows * es;
  const size_t norms = (size_t)(2 * sh.d + 2 * c.head_dim) * es, cache = (size_t)kvrows * c.max_pos * es;
  dec->off_wo = align256(wqkv);
  dec->off_norms = dec->off_wo + align256(wo);
  dec->off_k = dec->off_norms + align256(norms);
  dec->off_v = dec->off_k + align256(cache);
  dec->layer_bytes = dec->off_v + align256(cache);
  if (cudaSetDevice(sh.device) != cudaSuccess) {
    cudaGetLastError();
    delete dec;
    return dfail(nullptr, MOE_ERR_CUDA, "cudaSetDevice failed");
  }
  dec->layers.resize(sh.n_layers);
  for (DecLayer& ly : dec->layers) {
    if (cudaMalloc(&ly.mem, dec->layer_bytes) != cudaSuccess) {
      ly.mem = nullptr;
      free_decoder(dec);
      delete dec;
      return dfail(nullptr, MOE_ERR_OOM, "device memory for the attention weights and KV caches");
    }
    ly.wqkv = ly.mem;
    ly.wo = ly.mem + dec->off_wo;
    ly.norms = ly.mem + dec->off_norms;
    ly.K = ly.mem + dec->off_k;
    ly.V = ly.mem + dec->off_v;
  }
  const int64_t part = moe::attention_scratch_bound(c.n_heads, c.n_kv_heads, c.head_dim, c.max_pos);
  const size_t f4 = sizeof(float);
  const size_t o_a = align256((size_t)sh.d * f4), o_qkv = o_a + align256((size_t)sh.d * f4);
  const size_t o_q = o_qkv + align256((size_t)(qrows + 2 * kvrows) * f4), o_o = o_q + align256((size_t)qrows * f4);
  const size_t o_part = o_o + align256((size_t)qrows * f4), o_hid = o_part + align256((size_t)part * f4);
  const size_t o_mout = o_hid + align256((size_t)sh.n_layers * sh.d * es);
  const size_t total = o_mout + align256((size_t)sh.n_layers * sh.d * es);
  if (cudaMalloc(&dec->work, total) != cudaSuccess) {
    dec->work = nullptr;
    free_decoder(dec);
    delete dec;
    return dfail(nullptr, MOE_ERR_OOM, "device memory for the decoder's work buffers");
  }
  cudaMemset(dec->work, 0, total);
  dec->x = (float*)dec->work;
  dec->a = (float*)(dec->work + o_a);
  dec->qkv = (float*)(dec->work + o_qkv);
  dec->q = (float*)(dec->work + o_q);
  dec->o = (float*)(dec->work + o_o);
  dec->part = (float*)(dec->work + o_part);
  dec->hid = dec->work + o_hid;
  dec->mout = dec->work + o_mout;
  *out = dec;
  return MOE_OK;
}

moe_status moe_decoder_set_layer(moe_decoder* dec, int32_t layer, const void* wq, const void* wk, const void* wv,
                                 const void* wo, const void* norm_in, const void* norm_post, const void* norm_q,
                                 const void* norm_k) {
  if (!dec) return MOE_ERR_INVALID;
  if (layer < 0 || layer >= dec->shape.n_layers) return dfail(dec, MOE_ERR_INVALID, "layer out of range");
  if (!wq || !wk || !wv || !wo || !norm_in || !norm_post || !norm_q || !norm_k)
    return dfail(dec, MOE_ERR_INVALID, "NULL weight pointer");
  if (cudaSetDevice(dec->shape.device) != cudaSuccess) return dfail(dec, MOE_ERR_CUDA, "cudaSetDevice failed");
  DecLayer& ly = dec->layers[layer];
  const int64_t d = dec->shape.d, D = dec->cfg.head_dim, es = dec->es;
  uint8_t* wqkv = (uint8_t*)ly.wqkv;
  uint8_t* nrm = (uint8_t*)ly.norms;
  const struct {
    void* dst;
    const void* src;
    size_t bytes;
  } parts[] = {{wqkv, wq, (size_t)(dec->qrows * d * es)},
               {wqkv + dec->qrows * d * es, wk, (size_t)(dec->kvrows * d * es)},
               {wqkv + (dec->qrows + dec->kvrows) * d * es, wv, (size_t)(dec->kvrows * d * es)},
               {ly.wo, wo, (size_t)(d * dec->qrows * es)},
               {nrm, norm_in, (size_t)(d * es)},
               {nrm + d * es, norm_post, (size_t)(d * es)},
               {nrm + 2 * d * es, norm_q, (size_t)(D * es)},
               {nrm + (2 * d + D) * es, norm_k, (size_t)(D * es)}};
  for (const auto& p : parts)
    if (cudaMemcpy(p.dst, p.src, p.bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
      cudaGetLastError();
      return dfail(dec, MOE_ERR_CUDA, "copying the layer's weights to the device");
    }
  ly.set = true;
  return MOE_OK;
}

moe_status moe_decoder_set_cache(moe_decoder* dec, int32_t layer, const void* k, const void* v, int64_t n_pos) {
  if (!dec) return MOE_ERR_INVALID;
  if (layer < 0 || layer >= dec->shape.n_layers) return dfail(dec, MOE_ERR_INVALID, "layer out of range");
  if (n_pos < 0 || n_pos > dec->cfg.max_pos) return dfail(dec, MOE_ERR_INVALID, "n_pos must be in [0, max_pos]");
  if (n_pos > 0 && (!k || !v)) return dfail(dec, MOE_ERR_INVALID, "NULL cache pointer");
  if (cudaSetDevice(dec->shape.device) != cudaSuccess) return dfail(dec, MOE_ERR_CUDA, "cudaSetDevice failed");
  DecLayer& ly = dec->layers[layer];
  const size_t row = (size_t)dec->cfg.head_dim * dec->es;
  if (n_pos > 0) {
    for (int w = 0; w < 2; w++) {
      const cudaError_t e = cudaMemcpy2D(w ? ly.V : ly.K, row * dec->cfg.max_pos, w ? v : k, row * n_pos, row * n_pos,
                                         dec->cfg.n_kv_heads, cudaMemcpyHostToDevice);
      if (e != cudaSuccess) {
        cudaGetLastError();
        return dfail(dec, MOE_ERR_CUDA, "copying the KV cache prefix to the device");
      }
    }
  }
  ly.n_pos = n_pos;
  return MOE_OK;
}

moe_status moe_decoder_step(moe_decoder* dec, const void* x_in, float* x_out, float* layer_log, void* stream) {
  if (!dec) return MOE_ERR_INVALID;
  if (!x_in || !x_out) return dfail(dec, MOE_ERR_INVALID, "NULL x_in or x_out");
  for (int l = 0; l < dec->shape.n_layers; l++) {
    if (!dec->layers[l].set)
      return dfail(dec, MOE_ERR_NOT_REGISTERED, "attention weights of layer " + std::to_string(l) + " not set");
    if (dec->layers[l].n_pos != dec->layers[0].n_pos)
      return dfail(dec, MOE_ERR_INVALID, "the layers' KV caches hold different numbers of positions");
  }
  if (dec->layers[0].n_pos >= dec->cfg.max_pos) return dfail(dec, MOE_ERR_CAPACITY, "the KV cache is full");
  if (cudaSetDevice(dec->shape.device) != cudaSuccess) return dfail(dec, MOE_ERR_CUDA, "cudaSetDevice failed");
  cudaStream_t s = (cudaStream_t)stream;
  const moe_status st = dec->es == 4 ? run_step<float>(dec, x_in, x_out, layer_log, s)
                                     : run_step<__nv_bfloat16>(dec, x_in, x_out, layer_log, s);
  if (st != MOE_OK) return st;
  for (DecLayer& ly : dec->layers) ly.n_pos++;
  return MOE_OK;
}

int64_t moe_decoder_position(const moe_decoder* dec) { return dec ? dec->layers[0].n_pos : -1; }

const char* moe_decoder_last_error(const moe_decoder* dec) { return dec ? dec->err.c_str() : g_create_err.c_str(); }

void moe_decoder_destroy(moe_decoder* dec) {
  if (!dec) return;
  cudaSetDevice(dec->shape.device);
  cudaDeviceSynchronize();
  free_decoder(dec);
  delete dec;
}

}  // extern "C"
