// Library-internal hooks between translation units (not part of the C ABI): the chained decoder
// (decoder.cu) runs the MoE layer of a handle one layer at a time, and the decode attention
// (attention.cu) without the C entry point's argument checks.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "moe.h"

namespace moe {

// What the decoder needs to know about a MoE handle.
struct MoeShape {
  int32_t d, n_layers, top_k, n_experts, wdtype, adtype, device;
  bool device_batch1;  // device schedule with max_batch == 1 (the schedule the decoder drives)
};
bool moe_shape(const moe_handle* h, MoeShape* out);

// Layer `layer` of the current decode step of h on stream s: hidden and out are device
// [n_layers x d] in the activation dtype, of which row `layer` is read and written. Layer 0
// first checks that every router and expert is registered and reports a failure flagged by an
// earlier step; the call for the last layer completes the step. On failure the pool is emptied
// (as after a failed moe_decode_step) and h's last error says why.
moe_status moe_run_layer(moe_handle* h, const void* hidden, void* out, int32_t layer, cudaStream_t s);
const char* moe_error_text(const moe_handle* h);

// Grouped-query decode attention (attention.cu); shapes as for moe_attention_decode.
bool attention_shape_ok(int32_t n_heads, int32_t n_kv_heads, int32_t head_dim);
// Partial-result floats that serve attention_launch for every n_pos in [1, max_pos].
int64_t attention_scratch_bound(int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t max_pos);
cudaError_t attention_launch(int32_t cache_dtype, const float* q, const void* k_cache, const void* v_cache,
                             int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t max_pos, int64_t n_pos,
                             float* out, float* scratch, cudaStream_t s);

}  // namespace moe
