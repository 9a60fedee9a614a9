// Device-driven decode step: one cooperative persistent kernel runs every layer of a decode
// step (router, slot lookup + LRU, miss transfer, expert FFN, combine) with no host round trip.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace moe {

// One residency record, same layout as moe_trace_rec in include/moe.h.
struct TraceRec {
  int32_t step, layer, expert, kind, slot, evicted;
};

enum { STAT_HITS = 0, STAT_MISSES = 1, STAT_EVICTIONS = 2, STAT_LAYER_STEPS = 3, STAT_N = 4 };
// Layers per worker barrier of the lookahead kernel when the pool allows it (cap >= 2 x this x k).
constexpr int kLaGroupMax = 2;

enum { FERR_BARRIER_TIMEOUT = 1, FERR_BAD_ROUTE = 2, FERR_NO_VICTIM = 4, FERR_PIPE_TIMEOUT = 8 };
// Flags after which every CTA leaves the kernel at its next grid barrier.
constexpr int FERR_FATAL = FERR_BARRIER_TIMEOUT | FERR_PIPE_TIMEOUT;

struct FusedArgs {
  int L, E, k, d, I, renorm, wdtype;
  int l_begin, l_end;          // layers [l_begin, l_end) run in this launch; the launch that ends at
                               // layer L completes the decode step (a chained decoder launches one
                               // layer at a time, each after the attention that produces its input)
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
  unsigned long long* slot_key;// [cap]: replacement key of the resident expert (smallest = first victim),
                               // ~0 if free. LRU and rotary: (last use << 32) | global id. Router-guided:
                               // guided_key(E, rank, last use, global id)
  int32_t* n_used;             // slots handed out so far; [n_used, cap) are free
  int64_t* step;               // decode steps completed (clock = step * L + layer)
  // per-layer scratch (device)
  float* z;                    // [L][E] router logits of the current decode step
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
  int touch_shift;             // log2 of the stride of the translation-warming touches (12 = 4 KB; 0 = none)
  // Victim candidates: the k smallest slot keys of a full pool, ascending, found by CTA 0 during
  // phase C (off the critical path) for the next layer-step's phase S; cand[kMaxRanks] holds how
  // many are valid (0: phase S scans every slot).
  unsigned long long* cand;    // [kMaxRanks + 1]
  int may_evict;               // LRU or router-guided with cap < experts in the stack (else no victim
                               // search is needed)
  // Rotary slot-group policy (policy == 1): each slot's previous occupant, its inverse, the hand.
  int policy;                  // 0 LRU, 1 rotary, 2 router-guided
  int32_t* prior;              // [cap]: global id last evicted from the slot, -1 none
  int32_t* prior_slot_of;      // [L*E]: the slot whose previous occupant is the id, -1 none
  int32_t* hand;               // [1]
  // Router-guided policy (policy == 2): every expert's rank in its layer's latest routing
  // (0 = highest logit, ties to the lower id; E before the layer's first routing).
  int32_t* rank;               // [L*E]
  unsigned* plan_flag;         // clock of the last layer-step whose plan CTA 0 has published (0: none)
  // Exact layer lookahead (k_fused_la): the worker CTAs' arrival counters, one per parity of the
  // layer group, and their values at launch. The plan arrays then hold every layer's plan, [L][k].
  unsigned* wbar_count;        // [2]
  unsigned wbar_base[2];
  int la_group;                // layers per worker barrier (1 or kLaGroupMax; needs cap >= 2 la_group k)
  int la_skew;                 // 1: a group's down rows run after the next group's gate/up rows (needs
                               // cap >= 3 la_group k, or every expert resident, and u for 4 groups)
};

// Router-guided replacement key: the victim is the smallest key, i.e. the largest rank, then the
// most recent use, then the lowest global id. Fields: E - rank (9 bits), ~last use (32 bits),
// global id (23 bits; the host checks L * E < 2^23).
constexpr int kGuidedGidBits = 23;
__host__ __device__ __forceinline__ unsigned long long guided_key(int E, int rank, uint32_t last_use, int gid) {
  return ((unsigned long long)(uint32_t)(E - rank) << 55) | ((unsigned long long)(0xffffffffu - last_use) << 23) |
         (unsigned long long)(uint32_t)gid;
}
__host__ __device__ __forceinline__ uint32_t guided_key_last_use(unsigned long long key) {
  return 0xffffffffu - (uint32_t)((key >> 23) & 0xffffffffull);
}
__host__ __device__ __forceinline__ int slot_key_gid(unsigned long long key, int policy) {
  return policy == 2 ? (int)(key & ((1ull << kGuidedGidBits) - 1)) : (int)(uint32_t)(key & 0xffffffffull);
}

// Maximum co-resident CTAs for the fused kernel of this shape (0 if it cannot launch).
int fused_grid(int wdtype, int d, int I, int k);
cudaError_t launch_fused(const FusedArgs& a, int grid, cudaStream_t s);

// Exact layer lookahead at batch 1 under LRU (layers' inputs all given with the step): CTA 0 runs
// the lookup steps of every layer in order while the other CTAs compute. Needs cap >= 2 k (or
// every expert resident): then no miss takes the slot of an expert the previous layer-step used,
// whose down rows may still be running when the miss's bytes arrive. Same decisions, trace and
// outputs as k_fused.
int fused_la_grid(int wdtype, int d, int I, int k, int group);
cudaError_t launch_fused_la(const FusedArgs& a, int grid, cudaStream_t s);

// Batched decode step: B sequences per step, one cooperative kernel over all layers. Per layer
// the needed experts are the union of every sequence's top k; each needed expert is read once
// and applied to all the sequences routed to it (a grouped GEMV).
constexpr int kMaxBatch = 64;
constexpr int kBatchedEvictCap = 4096;  // slot counts this large or smaller can evict in a batched step
constexpr int kBatchedPhases = 6;       // router, top-k, select, gate-up, down, combine

struct BatchArgs {
  // Tensor-core variant (bf16 weights): TMA maps over the slot pool and over the pairs'
  // activations and u vectors in plan order (pairs grouped by expert, so an expert's pairs are
  // consecutive rows).
  CUtensorMap map_gu;          // pool gate/up rows: dims {d, 2I, cap}, box {64, 128, 1}, 128-B swizzle
  CUtensorMap map_d;           // pool W_d rows: dims {I, d, cap}, box {64, 128, 1}
  CUtensorMap map_x;           // xg: dims {d, Bmax*k}, box {64, 16}
  CUtensorMap map_u;           // ug: dims {I, Bmax*k}, box {64, 16}
  __nv_bfloat16* xg;           // [Bmax*k][d] activation of each pair, plan order
  __nv_bfloat16* ug;           // [Bmax*k][I] u of each pair, plan order
  int L, E, k, d, I, renorm, wdtype;
  int B;                       // sequences this step (<= Bmax)
  int Bmax;                    // row stride of the routing log
  BlobLayout lay;
  int64_t slot_stride;
  int64_t cap;
  int64_t n_gid;
  const uint8_t* routers;      // device [L][E][d]
  const void* hidden;          // device [L][B][d]
  void* out;                   // device [L][B][d]
  uint8_t* pool;
  const uint8_t* arena;
  int32_t* slot_of;
  unsigned long long* slot_key;
  int32_t* n_used;
  int64_t* step;
  // per-layer scratch
  float* z;                    // [L][Bmax][E] router logits of the current decode step
  int32_t* sel_e;              // [B*k] expert of pair p = b*k + r
  float* sel_g;                // [B*k] its gate
  int32_t* plan_n;             // [2] distinct experts needed this layer-step, and how many missed
  int32_t* plan_slot;          // [E] per needed expert: the misses (ascending id), then the hits
  int32_t* plan_gid;           // [E]
  int32_t* plan_miss;          // [E]
  int32_t* plan_off;           // [E] start of its pairs in plan_tok
  int32_t* plan_cnt;           // [E] number of pairs routed to it
  int32_t* plan_tok;           // [B*k] pair indices grouped by needed expert, ascending
  float* u;                    // [B*k][I]
  float* y;                    // [B*k][d]
  TraceRec* trace;
  int64_t trace_cap;
  unsigned long long* trace_n;
  int32_t* route_idx;          // [L][Bmax][k]
  float* route_gate;           // [L][Bmax][k]
  unsigned long long* stats;
  unsigned* bar_count;
  unsigned bar_base;
  int* err;
  unsigned long long barrier_timeout_ns;
  unsigned long long* phase_ts; // optional [L][kBatchedPhases] + 1
  unsigned* work;              // [2] work-item counters of phases C and D (reset in phase S)
  int touch_shift;             // log2 of the translation-warming touch stride (0: no touches)
  int tg_max;                  // pairs staged in shared memory at a time (batched_tg)
  int router_tb;               // sequences per router work item (batched_router_tb)
  int policy;                  // 0 LRU, 1 rotary, 2 router-guided
  int32_t* rank;               // [L*E] router-guided: rank in the layer's latest routing (best over the batch)
  int32_t* rank_best;          // [E] router-guided scratch: this layer-step's best rank over the batch
  // Rotary slot-group policy (policy == 1), as in FusedArgs
  int32_t* prior;              // [cap]
  int32_t* prior_slot_of;      // [n_gid]
  int32_t* hand;               // [1]
};

// Pairs staged per group for this shape, and the co-resident grid (0: shape or cap unsupported).
int batched_tg(int wdtype, int d, int I);
// Sequences per router work item (1..8: their activations fit in the kernel's shared memory).
int batched_router_tb(int wdtype, int d, int I, bool tensor_cores);
int fused_batched_grid(int wdtype, int d, int I, int64_t cap, int64_t n_gid);
cudaError_t launch_fused_batched(const BatchArgs& a, int grid, cudaStream_t s);

// Tensor-core variant: bf16 weights, d a multiple of 128 and I of 64. Seven phases per layer
// (router, top-k, select, gather, gate-up, down, combine).
constexpr int kBatchedTcPhases = 7;
bool batched_tc_supported(int wdtype, int d, int I);
int fused_batched_tc_grid(int d, int I, int64_t cap, int64_t n_gid);
cudaError_t launch_fused_batched_tc(const BatchArgs& a, int grid, cudaStream_t s);

}  // namespace moe
