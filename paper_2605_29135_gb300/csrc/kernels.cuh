// Device kernels of the capped-residency MoE decode step and their launch wrappers.
//
// Slot layout of one expert (a slot holds exactly this byte image; the host arena keeps the
// same image per expert so a miss is one contiguous copy):
//   [GU rows]   for i in 0..I-1: gate row i (d elements) then up row i (d elements)
//   [GU scales] int4 only: for i in 0..I-1: gate scales of row i (d/128 bf16), up scales of row i
//   [D rows]    W_d rows o = 0..d-1 (I elements each)
//   [D scales]  int4 only: W_d scales, row-major [d x I/128] bf16
// Element storage: fp32, bf16, or int4 (two's-complement nibbles, element 2j in the low nibble
// of byte j of its row). Activations are fp32 with fp32 weights and bf16 otherwise.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace moe {

enum { WD_FP32 = 0, WD_BF16 = 1, WD_INT4 = 2 };

struct BlobLayout {
  int64_t row_bytes_gu;    // bytes of one gate (or up) row
  int64_t row_bytes_d;     // bytes of one W_d row
  int64_t gu_scale_off;    // int4: offset of the GU scales region
  int64_t d_off;           // offset of the W_d rows region
  int64_t d_scale_off;     // int4: offset of the W_d scales region
  int64_t total;           // bytes of the expert image
};

BlobLayout make_layout(int wdtype, int64_t d, int64_t I);

constexpr int kMaxRanks = 16;

// u_t = silu(W_g x) * (W_u x) for the experts in blob[0..n_tasks), all on the same input x.
struct GateUpArgs {
  int n_tasks;
  int d, I;
  BlobLayout lay;
  const void* x;                   // [d] activations (fp32 with fp32 weights, else bf16)
  const uint8_t* blob[kMaxRanks];  // expert images in their slots
  float* u[kMaxRanks];             // outputs [I] fp32
};

// out = sum_r gate[r] * (W_d^(r) u_r), ranks in order.
struct DownArgs {
  int k;
  int d, I;
  BlobLayout lay;
  const uint8_t* blob[kMaxRanks];  // expert images in rank order
  float gate[kMaxRanks];
  const float* u;                  // [k x I] fp32, rank-major
  void* out;                       // [d] activations
};

// Routing result as written by the router kernel into host-mapped memory.
struct RouteOut {
  int32_t idx[kMaxRanks];
  float gate[kMaxRanks];
  float z[256];          // the logits, when RouterArgs::want_z (router-guided policy)
  volatile int64_t seq;  // written last, after a system-scope fence
};

struct RouterArgs {
  const void* w;      // W_r [E x d] device (fp32 or bf16)
  const void* h;      // hidden [d]
  int E, d, k, renorm;
  int wdtype;         // WD_FP32 or WD_BF16
  RouteOut* out;      // device address of host-mapped memory
  int64_t seq;
  int want_z;         // also publish the E logits
};

cudaError_t launch_router(const RouterArgs& a, cudaStream_t s);
// One 4-byte read from the SMs of every (1 << shift)-byte page of [base, base + bytes), base a
// device address of page-locked host memory (the host tier).
cudaError_t launch_touch_pages(const uint8_t* base, int64_t bytes, int shift, cudaStream_t s);
cudaError_t launch_gateup(const GateUpArgs& a, int wdtype, cudaStream_t s);
cudaError_t launch_down_combine(const DownArgs& a, int wdtype, cudaStream_t s);

}  // namespace moe
