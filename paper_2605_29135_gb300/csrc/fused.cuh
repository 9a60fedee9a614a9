// Device-driven decode step: one cooperative persistent kernel runs every layer of a decode
// step (router, slot lookup + LRU, miss transfer, expert FFN, combine) with no host round trip.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace moe {

// One residency record, same layout as moe_trace_rec in include/moe.h.
struct TraceRec {
  int32_t step, layer, expert, kind, slot, evicted;
};

enum { STAT_HITS = 0, STAT_MISSES = 1, STAT_EVICTIONS = 2, STAT_LAYER_STEPS = 3, STAT_N = 4 };
enum { FERR_BARRIER_TIMEOUT = 1, FERR_BAD_ROUTE = 2, FERR_NO_VICTIM = 4 };

struct FusedArgs {
  int L, E, k, d, I, renorm, wdtype;
  BlobLayout lay;
  int64_t slot_stride;
  int64_t cap;
  const uint8_t* routers;      // device [L][E][d] (fp32 or bf16)
  const void* hidden;          // device [L][d]
  void* out;                   // device [L][d]
  uint8_t* pool;               // device slot pool
  const uint8_t* arena;        // host tier (device-accessible address of page-locked host memory)
  // residency state (device): lookup table and recency
  int32_t* slot_of;            // [L*E], -1 if not resident
  unsigned long long* slot_key;// [cap]: (last use << 32) | global id of the resident expert; ~0 if free
  int32_t* n_used;             // slots handed out so far; [n_used, cap) are free
  int64_t* step;               // decode steps completed (clock = step * L + layer)
  // per-layer scratch (device)
  float* z;                    // [E] router logits
  int32_t* plan_slot;          // [k] slot of rank r
  int32_t* plan_gid;           // [k] global expert id of rank r
  int32_t* plan_miss;          // [k] 1 if rank r was a miss this layer-step
  float* plan_gate;            // [k]
  float* u;                    // [k][I]
  // outputs (device)
  TraceRec* trace;             // [trace_cap]
  int64_t trace_cap;
  unsigned long long* trace_n; // records produced (stored while < trace_cap)
  int32_t* route_idx;          // [L][k] routing of the last step
  float* route_gate;           // [L][k]
  unsigned long long* stats;   // [STAT_N]
  unsigned* bar_count;         // monotonic arrival counter of the grid barriers (wraps mod 2^32)
  unsigned bar_base;           // its value when this launch starts
  int* err;                    // FERR_* flags, sticky until the host clears them
  unsigned long long barrier_timeout_ns;
  unsigned long long* phase_ts; // optional [L][4]: global-timer ns at the end of phases R, S, C, D
                                // (CTA 0, after each barrier); NULL = off
  int miss_ctas;               // CTAs that stream missed experts from the host tier in phase C
  int touch_shift;             // log2 of the stride of the translation-warming touches (12 = 4 KB)
};

// Maximum co-resident CTAs for the fused kernel of this shape (0 if it cannot launch).
int fused_grid(int wdtype, int d, int I, int k);
cudaError_t launch_fused(const FusedArgs& a, int grid, cudaStream_t s);

}  // namespace moe
