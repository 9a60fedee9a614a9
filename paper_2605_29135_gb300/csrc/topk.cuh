// Warp-level router selection shared by the decode kernels: top k of one row of E <= 256 logits
// with ties going to the lower expert id, then the gates (softmax over the selected logits when
// renormalising, else the full-softmax probability of each selected expert).
#pragma once
#include <math.h>

#include "dev.cuh"

namespace moe {
namespace dev {

// One warp, all lanes. z: the row's E logits (global memory, read through L2). Lane r < k gets
// rank r: its expert id in out_i and its gate in out_g; lanes >= k get -1 and 0.
__device__ __forceinline__ void warp_topk(const float* z, int E, int k, int renorm, int lane, int& out_i,
                                          float& out_g) {
  constexpr int PER = 8;  // E <= 256
  uint32_t key[PER];
#pragma unroll
  for (int j = 0; j < PER; j++) {
    const int e = j * 32 + lane;
    key[j] = e < E ? ord_key(__ldcg(z + e)) : 0u;
  }
  float my_z = 0.f;
  int my_i = -1;
  for (int r = 0; r < k; r++) {
    uint32_t bk = 0u;
    int bi = 0x7fffffff;
#pragma unroll
    for (int j = 0; j < PER; j++) {
      if (key[j] > bk) {
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
  const float ex = lane < k ? expf(my_z - m) : 0.f;
  float denom;
  if (renorm) {
    denom = warp_sum(ex);
  } else {
    float part = 0.f;
    for (int e = lane; e < E; e += 32) part += expf(__ldcg(z + e) - m);
    denom = warp_sum(part);
  }
  out_i = lane < k ? my_i : -1;
  out_g = lane < k ? ex / denom : 0.f;
}

}  // namespace dev
}  // namespace moe
