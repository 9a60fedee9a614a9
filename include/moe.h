/*
 * moe.h -- C ABI of the GB300 capped-residency MoE decode library (libmoe.so).
 *
 * One decode step of a stack of Mixture-of-Experts layers whose experts do not
 * all fit in GPU memory. This is the residency problem of the paper (Section
 * "Rotary GPU Concept", Fig. 1): full expert weights stay in a host memory
 * tier; a fixed-capacity group of accelerator slots holds a subset of the
 * experts; a lookup table maps expert id -> slot; the routing result (hidden
 * state h, routing vector r) drives selective loads into slots and evictions
 * from them. The paper does not disclose its replacement policy; this library
 * uses a deterministic LRU with ties broken toward the lower global expert id.
 *
 * Per layer, in order (layers are processed strictly one after another and a
 * layer never looks at a later layer's input):
 *   1. router: z = W_r h (fp32 accumulation), top-k by z (ties -> lower id),
 *      gates g_r = softmax over the k selected logits (= p_{e_r} / sum_j p_{e_j});
 *   2. slot lookup + LRU: hit -> slot; miss -> lowest free slot, else evict the
 *      unpinned resident with the smallest (last use, global id);
 *   3. misses are copied from the pinned host arena into their slots on an
 *      internal copy stream, overlapped with the hit experts' compute;
 *   4. SwiGLU expert FFN from the slots: u = silu(W_g x) * (W_u x), y_r = W_d u
 *      (fp32 u and y; int4 weights dequantised in registers);
 *   5. out = sum_r g_r y_r in rank order (deterministic).
 *
 * Conventions
 *   - Every call returns a moe_status; nothing is thrown across the ABI.
 *     moe_last_error() gives a message for the last failure on a handle.
 *   - Pointers are host pointers unless a parameter says "device".
 *   - Ownership: the library owns everything it allocates; register/set calls
 *     copy the caller's buffers, which may be freed afterwards.
 *   - Threading: one handle is used by one host thread at a time, except that
 *     moe_register_host_experts may be called concurrently for distinct
 *     (layer, expert) pairs.
 *   - Device: the handle is bound to cfg.device; calls set that device.
 */
#ifndef MOE_H_
#define MOE_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct moe_handle moe_handle;

typedef enum {
  MOE_OK = 0,
  MOE_ERR_INVALID = -1,        /* bad argument or configuration */
  MOE_ERR_OOM = -2,            /* device or pinned host allocation failed */
  MOE_ERR_CUDA = -3,           /* a CUDA runtime call failed */
  MOE_ERR_CAPACITY = -4,       /* slot cap below one layer-step's working set */
  MOE_ERR_NOT_REGISTERED = -5, /* a router or expert needed by the step was never registered */
  MOE_ERR_TIMEOUT = -6,        /* a bounded wait for the device ran out */
  MOE_ERR_TRACE_OVERFLOW = -7  /* residency records were dropped (trace buffer full) */
} moe_status;

/* Storage types (wdtype: expert weights; adtype: activations hidden/out). */
enum {
  MOE_DTYPE_FP32 = 0,
  MOE_DTYPE_BF16 = 1,
  MOE_DTYPE_INT4_G128 = 2 /* symmetric int4, groups of 128 along the input dim, bf16 scales */
};

/* How a decode step is scheduled (both compute the same results and the same residency trace).
 *   MOE_SCHEDULE_DEVICE: one cooperative persistent kernel per decode step runs every layer. The
 *     lookup table lives in device memory and is updated by the kernel; a missed expert is
 *     streamed from the page-locked host tier over the host link by the warps that use it,
 *     stored into its freed slot and used in the same pass, concurrently with the hit experts'
 *     compute. moe_decode_step returns right after the launch (fully asynchronous).
 *   MOE_SCHEDULE_HOST_COPY_ENGINE: per layer, the routing result is published to mapped host
 *     memory, the host updates the lookup table and issues one cudaMemcpyAsync per miss on an
 *     internal copy stream; the hit experts' kernels run while the copies are in flight and
 *     each missed expert's kernels wait for its copy. moe_decode_step blocks once per layer.
 * Batched decoding (max_batch > 1, device schedule only; the paper describes batch-1 decoding and
 * has no counterpart): per layer the needed experts are the union of the batch's top-k choices,
 * one lookup-table step runs for that union (one record per distinct expert, ascending id), and
 * each needed expert is read once and applied to every sequence routed to it. */
enum { MOE_SCHEDULE_DEVICE = 0, MOE_SCHEDULE_HOST_COPY_ENGINE = 1 };

/* Expert FFN of batched steps (max_batch > 1).
 *   MOE_BATCHED_AUTO: tensor cores when the shape allows (bf16 weights, d a multiple of 128,
 *     d_ff of 64): per layer-step each needed expert's gate/up and down matrices are multiplied
 *     with the stacked activations of the pairs routed to it (tcgen05 MMA, operands streamed by
 *     TMA, fp32 accumulation; u is rounded to bf16 between the two projections). Missed experts
 *     are first copied into their slots, so hits and misses share the arithmetic. Other shapes:
 *     CUDA cores, as MOE_BATCHED_CUDA_CORES.
 *   MOE_BATCHED_CUDA_CORES: grouped GEMV on CUDA cores (fp32 accumulation, fp32 u); missed
 *     experts stream from the host tier straight into their slot and the compute. */
enum { MOE_BATCHED_AUTO = 0, MOE_BATCHED_CUDA_CORES = 1 };

/* Replacement policy of the slot group.
 *   MOE_POLICY_LRU (default): misses take the lowest free slot, else evict the resident expert not
 *     needed this layer-step with the smallest (last use, global id). Both schedules.
 *   MOE_POLICY_ROTARY: this library's reading of the paper's rotary slot group (Fig. 1, Fig. 2;
 *     the paper gives no algorithm). The slots form a ring with a hand and each slot remembers its
 *     previous occupant. A miss returns to the slot it was last evicted from when that slot holds no
 *     expert of the layer-step (reverse rotation), else takes the first such slot at or after the
 *     hand, which then moves past it (forward rotation). Hits change nothing. Misses in ascending
 *     global id. Both schedules; a batched step (device schedule) applies it to the union of the
 *     batch's experts. */
/*   MOE_POLICY_GUIDED: router-guided replacement, one reading of the paper's residency decisions
 *     that use information produced during execution (Sec. 3). Each layer keeps the rank of every
 *     expert in its most recent routing (0 = highest logit; for a batch, the best rank over its
 *     sequences). A miss takes the lowest free slot, else evicts the resident not needed this
 *     layer-step with the largest rank, ties to the more recent use, then to the lower global id.
 *     Both schedules (device: n_layers * n_experts < 2^23), and the residency planner. */
enum { MOE_POLICY_LRU = 0, MOE_POLICY_ROTARY = 1, MOE_POLICY_GUIDED = 2 };

typedef struct {
  int32_t d;          /* hidden size */
  int32_t n_experts;  /* experts per layer, E (<= 256) */
  int32_t top_k;      /* experts per token, k (<= 16, <= E) */
  int32_t d_ff;       /* SwiGLU intermediate size, I */
  int32_t n_layers;   /* L */
  int32_t max_batch;  /* most sequences per decode step, 1..64. Above 1 needs MOE_SCHEDULE_DEVICE, and a
                         cap that can evict (cap < n_layers * n_experts) must be at most 4096 slots */
  int32_t wdtype;     /* MOE_DTYPE_FP32 (needs adtype FP32), BF16 or INT4_G128 (need adtype BF16) */
  int32_t adtype;     /* MOE_DTYPE_FP32 or MOE_DTYPE_BF16 */
  int64_t cap_slots;  /* expert slots on the device; 0 => floor(cap_bytes / expert bytes) */
  int64_t cap_bytes;  /* device expert-pool budget in bytes (used when cap_slots == 0) */
  int32_t renorm;     /* 1: gates renormalised over the top k (default); 0: raw softmax probabilities */
  int32_t device;     /* CUDA device ordinal */
  void* device_pool;  /* optional caller-owned device buffer of >= moe_pool_bytes(cfg) bytes, 256-B aligned;
                         NULL => the library allocates the pool */
  int64_t trace_capacity; /* residency records kept (device buffer for MOE_SCHEDULE_DEVICE, host otherwise);
                             0 disables the trace */
  int32_t schedule;       /* MOE_SCHEDULE_DEVICE (default) or MOE_SCHEDULE_HOST_COPY_ENGINE */
  int32_t miss_ctas;      /* MOE_SCHEDULE_DEVICE, max_batch 1: CTAs that stream missed experts over the
                             host link while the others compute the hits (0: library default). Batched
                             steps hand work items to all CTAs, missed experts first, and ignore it */
  int32_t batched_path;   /* MOE_BATCHED_AUTO (default) or MOE_BATCHED_CUDA_CORES */
  int32_t policy;         /* MOE_POLICY_LRU (default), MOE_POLICY_ROTARY or MOE_POLICY_GUIDED */
  int32_t lookahead;      /* 1: exact layer lookahead (the layers' inputs are all given with the step, so the
                             decisions, the trace and the outputs are those of 0). MOE_SCHEDULE_HOST_COPY_ENGINE:
                             route layer l + 1 as soon as layer l's routing has reached the host, and issue its
                             miss copies while layer l computes; a copy into a slot layer l still reads waits
                             for layer l's kernels. MOE_SCHEDULE_DEVICE (max_batch 1, MOE_POLICY_LRU): one kernel
                             routes every layer first, then CTA 0 runs the layers' lookups in order ahead of
                             the other CTAs, which compute the layers in groups (two layers per group from
                             4 * top_k slots on), arriving on a counter after each group's gate/up rows;
                             from 3 * top_k slots per layer of a group, or with every expert resident, a
                             group's down rows run after the next group's gate/up rows. Needs cap_slots >=
                             2 * top_k unless every expert is resident. Steps of a
                             chained decoder (moe_decoder_step) run layer by layer whatever this says.
                             0 (default): one layer after another. */
} moe_config;

/* One residency record: a requested expert's outcome in one layer-step. */
typedef struct {
  int32_t step;    /* decode step index since create/reset */
  int32_t layer;
  int32_t expert;  /* expert id within the layer */
  int32_t kind;    /* 0 hit, 1 miss, 2 prefetch admission (residency planner only) */
  int32_t slot;    /* slot holding the expert after the step */
  int32_t evicted; /* global id (layer * E + expert) of the evicted expert; -1 if none */
} moe_trace_rec;

typedef struct {
  int64_t steps;       /* decode steps run */
  int64_t layer_steps; /* layer-steps run */
  int64_t hits;
  int64_t misses;
  int64_t evictions;
  int64_t miss_bytes;  /* bytes copied host -> device for misses */
} moe_stats;

/* Per-kernel-class timing gathered with CUDA events on the launching streams while
 * profiling is on (see moe_profile_enable). */
typedef struct {
  char name[32];
  int64_t launches;
  double total_ms;
  int64_t bytes;       /* algorithmic bytes moved by all launches (weights read + vectors read/written) */
} moe_kernel_time;

/* Bytes of one expert's weights as stored in a slot (scales included for int4). */
int64_t moe_expert_bytes(const moe_config* cfg);
/* Bytes the device expert pool needs for cfg (slots * 256-B aligned slot stride), or < 0 if cfg is invalid. */
int64_t moe_pool_bytes(const moe_config* cfg);

/* Paper: the fixed slot group and its capacity (Sec. "Rotary GPU Concept", Fig. 1 "Rotary Slot
 * Group"); the capacity error is the clean form of the start-up failure of Sec. "Failure Analysis".
 * Validate cfg, allocate the device pool (unless cfg->device_pool is given), the pinned host
 * arena for all n_layers * n_experts experts, router storage and work buffers.
 * MOE_ERR_CAPACITY if the slot count is below min(E, k * max_batch), the most distinct experts
 * one layer-step can need (a clean failure instead of a start-up that cannot run).
 * On failure *out is NULL and nothing stays allocated. */
moe_status moe_create(const moe_config* cfg, moe_handle** out);

/* Paper: the router whose output is Fig. 1's "Routing Result" (Sec. "Rotary GPU Concept").
 * Router weights of one layer: W_r [E x d] row-major, host memory, fp32 when wdtype is FP32,
 * else bf16. Copied to device memory (routers are always resident, outside the slot cap). */
moe_status moe_set_router(moe_handle* h, int32_t layer, const void* w_r);

/* Paper: Fig. 1 "Host Memory / Storage Tier", the full weights kept outside the accelerator
 * (Sec. "Rotary GPU Concept").
 * One expert's weights into the pinned host tier (the paper's host memory tier). Row-major,
 * out x in: w_gate [I x d], w_up [I x d], w_down [d x I].
 *   FP32/BF16: elements of that type.
 *   INT4_G128: packed nibbles, byte j of a row = element 2j (low nibble) and 2j+1 (high),
 *              two's complement; `scales` = bf16 [I x d/128] (gate) ++ [I x d/128] (up)
 *              ++ [d x I/128] (down). NULL otherwise.
 * The weights are repacked into the slot layout. If the expert is resident its slot copy is
 * NOT refreshed; call moe_reset_residency after re-registering resident experts. */
moe_status moe_register_host_experts(moe_handle* h, int32_t layer, int32_t expert, const void* w_gate,
                                     const void* w_up, const void* w_down, const void* scales);

/* Paper: Fig. 1's cycle, routing result -> lookup table -> selective load into slots / evict
 * (Sec. "Rotary GPU Concept"), run once per layer of a decode step.
 * One decode step over all layers for `batch` sequences (1 <= batch <= max_batch; MOE_ERR_INVALID
 * otherwise). hidden: device [n_layers x batch x d] (adtype), the input of every layer; out:
 * device [n_layers x batch x d] (adtype); both 16-byte aligned (MOE_ERR_INVALID otherwise, before
 * any launch). Work is ordered on `stream`
 * (a cudaStream_t; NULL = legacy default stream). hidden must stay valid and out must not be
 * read until `stream` reaches the end of the step. Calls on one handle must use one stream or
 * be serialised by the caller.
 *   MOE_SCHEDULE_DEVICE: enqueues one kernel and returns. The first step after creation, a reset
 *     or a gap of 2 s or more since the previous step's launch (with a pool smaller than the
 *     stack) first enqueues one read per 4 KB page of the host tier from all SMs: after an idle
 *     gap the host link's first reads run 2-3x slower for ~1 s of streaming, and this pass pays
 *     that cost once (about 0.5-0.7 s for a 58 GB tier) instead of over the next ~100 steps.
 *     A failure detected on the device
 *     (a grid barrier that timed out, an invalid routing result) is reported by the next call
 *     on the handle that synchronises (decode_step, get_stats, get_residency_trace, ...), as
 *     MOE_ERR_TIMEOUT or MOE_ERR_CUDA, and empties the pool.
 *   MOE_SCHEDULE_HOST_COPY_ENGINE: blocks once per layer until that layer's routing result has
 *     reached the host (bounded wait, MOE_ERR_TIMEOUT) and returns once the last layer's work
 *     is enqueued.
 * If a CUDA call fails mid-step the residency state is reset (empty pool) and MOE_ERR_CUDA is
 * returned. */
moe_status moe_decode_step(moe_handle* h, const void* hidden, void* out, int32_t batch, void* stream);

/* Paper: as moe_decode_step (Fig. 1), with the step's activations in host memory.
 * moe_decode_step on host buffers (pinned or pageable): copies hidden to the device, runs the
 * step on an internal stream, copies out back and waits for completion. */
moe_status moe_decode_step_host(moe_handle* h, const void* hidden_host, void* out_host, int32_t batch);

/* Paper: the history of Fig. 1's "Lookup Table" (sub-module id -> slot position) and of the
 * selective loads and evictions behind it (Sec. "Rotary GPU Concept").
 * Copy residency records [start, start + cap) of the trace into buf. *n_copied = records copied,
 * *n_total = records kept. MOE_ERR_TRACE_OVERFLOW (after copying) if records were dropped. */
moe_status moe_get_residency_trace(moe_handle* h, int64_t start, moe_trace_rec* buf, int64_t cap,
                                   int64_t* n_copied, int64_t* n_total);

/* Paper: Fig. 1 "Routing Result" (routing vector r) of the last step.
 * Routing of the last decode step: idx int32 [n_layers x max_batch x k], gate fp32 [same]; n is
 * the entries buf can hold (MOE_ERR_INVALID if below n_layers * max_batch * k). Rows b >= the last
 * step's batch are stale. */
moe_status moe_get_last_routing(moe_handle* h, int32_t* idx, float* gate, int64_t n);

/* Paper: the counts of Fig. 1's selective loads and evictions (Sec. "Rotary GPU Concept"); the
 * transfer cost the Discussion names is miss_bytes. MOE_SCHEDULE_DEVICE: waits for the handle's
 * outstanding steps. */
moe_status moe_get_stats(moe_handle* h, moe_stats* out);

/* Router logits of the last decode step, fp32 [n_layers x max_batch x n_experts] (z = W_r h as the
 * device computed it; the router-guided policy ranks experts by them; rows b >= the step's batch
 * are stale). MOE_SCHEDULE_DEVICE, or MOE_SCHEDULE_HOST_COPY_ENGINE under MOE_POLICY_GUIDED
 * (MOE_ERR_INVALID otherwise, or if n is below n_layers * max_batch * n_experts). Waits for the
 * step. */
moe_status moe_get_last_logits(moe_handle* h, float* z, int64_t n);

/* Paper: the slot group of Fig. 1 emptied (every sub-module back in the host tier only).
 * Empty the slot pool (all experts non-resident), step clock 0, trace and stats cleared. */
moe_status moe_reset_residency(moe_handle* h);

/* Paper: Fig. 1 "selective load" ahead of the first step (a warm slot group).
 * Warm start: copy experts into free slots in ascending global id order until the pool is full
 * (with cap_slots >= n_layers * n_experts every expert becomes resident). Preloaded experts count
 * as used before every decode step, so they are the first victims; the copies are not residency
 * records and do not change the stats. Synchronous; *n_loaded (optional) = experts copied. */
moe_status moe_preload(moe_handle* h, int64_t* n_loaded);

/* Profiling: with on = 1, every kernel launch and miss copy of later steps is bracketed by
 * CUDA events on its stream. moe_profile_read waits for the recorded work, then reports one
 * entry per kernel class (router, gateup, down_combine, miss_copy, fused_step) and, for the
 * device schedule, per phase of the fused kernel (fused_phase_router, _select, _gateup, _down;
 * for batches also _topk and _combine, and _gather in the tensor-core variant: per layer-step
 * durations from the kernel's global timer), accumulated since the last read, and clears the
 * accumulators. */
moe_status moe_profile_enable(moe_handle* h, int32_t on);
moe_status moe_profile_read(moe_handle* h, moe_kernel_time* out, int32_t cap, int32_t* n_out);

/* ---- Fault injection (test hook; the paper has no counterpart) --------------------------------
 * Arms one fault for the next decode step, to exercise the error paths without faulting a GPU:
 *   MOE_FAULT_BARRIER_TIMEOUT (device schedule): the step's grid barriers wait for an arrival
 *     count no launch reaches, with a 0.2 s limit. Every wait runs out, the kernel exits, and the
 *     step (or the next call that synchronises) returns MOE_ERR_TIMEOUT with the pool emptied.
 *   MOE_FAULT_COPY_ERROR (host copy-engine schedule): the step's first miss copy reports a CUDA
 *     error before it is issued; the step returns MOE_ERR_CUDA with the pool emptied.
 *   MOE_FAULT_NONE disarms. MOE_ERR_INVALID for a kind the handle's schedule cannot take. */
enum { MOE_FAULT_NONE = 0, MOE_FAULT_BARRIER_TIMEOUT = 1, MOE_FAULT_COPY_ERROR = 2 };
moe_status moe_inject_fault(moe_handle* h, int32_t kind);

/* ---- Allocation-free routing --------------------------------------------------------------
 * The paper has no counterpart to this call; it exists for callers that cannot allocate device
 * memory at the point where they route (an inference runtime that reserves all device memory at
 * start-up and forbids later cudaMalloc, a plug-in that runs inside a host process owning the
 * allocator, code running under a lock that allocation would need). It needs no handle.
 *
 * Router GEMV + top-k + gates for `rows` hidden vectors against one router matrix, with the same
 * arithmetic as the router stage of moe_decode_step: z = W_r h (fp32 accumulation), top-k by z
 * (ties -> lower id), gates = softmax over the k selected logits (renorm = 1) or the
 * full-softmax probabilities (renorm = 0).
 *   w_r     device, [n_experts x d] row-major, fp32 (wdtype MOE_DTYPE_FP32) or bf16 (MOE_DTYPE_BF16)
 *   hidden  device, [rows x d], same element type as w_r
 *   idx     device output, int32 [rows x top_k], expert ids in descending logit order
 *   gate    device output, fp32 [rows x top_k]
 *   stream  cudaStream_t the two kernels are ordered on (NULL = legacy default stream)
 * The logits go to a fixed scratch array of MOE_NOALLOC_MAX_ROWS * MOE_NOALLOC_MAX_EXPERTS floats
 * (64 KiB) inside the library, held on every device that loads the library until the process
 * exits; no memory is allocated by the call. The first call on a device looks up that array's
 * device address (cudaGetSymbolAddress), so make the first call on each device before any stream
 * capture. Every call reuses the same array: calls whose work overlaps on the GPU (different
 * streams or host threads) race on it and must be serialised by the caller.
 * Returns MOE_ERR_CAPACITY if rows > MOE_NOALLOC_MAX_ROWS or n_experts > MOE_NOALLOC_MAX_EXPERTS,
 * MOE_ERR_INVALID for other bad arguments (top_k > 16 or > n_experts, d * element bytes not a
 * multiple of 16 or above 48 KiB, NULL pointers, w_r or hidden not 16-byte aligned, idx or gate
 * not 4-byte aligned), MOE_ERR_CUDA if a launch fails. Every argument check runs before any CUDA
 * call. A logit that is NaN still yields expert ids inside [0, n_experts). */
#define MOE_NOALLOC_MAX_ROWS 64
#define MOE_NOALLOC_MAX_EXPERTS 256
moe_status moe_route_noalloc(const void* w_r, const void* hidden, int32_t rows, int32_t n_experts, int32_t d,
                             int32_t top_k, int32_t renorm, int32_t wdtype, int32_t* idx, float* gate, void* stream);

/* ---- Attention of the decoder block around the MoE layer ------------------------------------
 * Grouped-query attention of one decode token over a KV cache (the decoder the paper ran kept a
 * 4096-token context). No handle; nothing is allocated.
 *   q        device fp32 [n_heads x head_dim], already normalised, rotated (scale 1/sqrt(head_dim)
 *            is applied inside)
 *   k_cache, v_cache  device [n_kv_heads x max_pos x head_dim] of cache_dtype (MOE_DTYPE_BF16 or
 *            MOE_DTYPE_FP32), 16-byte aligned; positions [0, n_pos) are read
 *   out      device fp32 [n_heads x head_dim]: query head h reads kv head h / (n_heads / n_kv_heads);
 *            out_h = sum_j softmax_j(q_h . k_j / sqrt(head_dim)) v_j
 *   scratch  device fp32 of at least moe_attention_scratch_floats(...) floats (per-split partials)
 *   stream   cudaStream_t the two kernels are ordered on (NULL = legacy default stream)
 * head_dim 64 or 128; n_heads / n_kv_heads in {1, 2, 4, 8}; 1 <= n_pos <= max_pos. MOE_ERR_INVALID
 * for other arguments (moe_attention_scratch_floats returns -1 for them), MOE_ERR_CUDA if a
 * launch fails. */
int64_t moe_attention_scratch_floats(int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t n_pos);
moe_status moe_attention_decode(const float* q, const void* k_cache, const void* v_cache, int32_t cache_dtype,
                                int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int64_t max_pos, int64_t n_pos,
                                float* out, float* scratch, int64_t scratch_floats, void* stream);

/* ---- Chained decoder blocks around the MoE layer ---------------------------------------------
 * One decode token at batch 1 through a stack of decoder blocks whose layers feed one another:
 * the paper's end-to-end setting (a whole MoE decoder at a 4096-token context, Sec.
 * "Experimental Setup"). The paper prints no architecture; the block is a Qwen3-MoE-class
 * reading. Per layer l, with the residual stream x (fp32) at position p:
 *   a = RMSNorm(x) * w_in;  q = W_q a [n_heads x head_dim];  k = W_k a, v = W_v a [n_kv_heads x head_dim]
 *   q_h = RoPE(RMSNorm(q_h) * w_q, p);  k_g = RoPE(RMSNorm(k_g) * w_k, p);  (k_g, v_g) -> cache row p
 *   o_h = sum_j softmax_j(q_h . K_j / sqrt(head_dim)) V_j over rows 0..p of kv head h / (n_heads / n_kv_heads)
 *   x += W_o [o_0 .. o_{n_heads-1}];  m = RMSNorm(x) * w_post;  x += MoE_l(m)
 * RMSNorm(y) = y / sqrt(mean(y^2) + eps); RoPE rotates element i with element i + head_dim/2 by
 * the angle p * rope_theta^(-2i/head_dim). MoE_l is layer l of the handle's decode step (routing,
 * one residency step of its slot group, expert FFN, combine); layer l + 1 routes on what layer l
 * produced, so every layer's MoE runs after its own attention.
 *
 * moe_decoder_create: moe must use MOE_SCHEDULE_DEVICE with max_batch 1, and outlives the
 *   decoder. Decode steps of the decoder advance the handle's decode steps, trace, statistics and
 *   slot group like moe_decode_step does (one decode step per token). Weights, KV caches and the
 *   MoE layers' inputs and outputs use the handle's activation storage: fp32 (MOE_DTYPE_FP32
 *   experts) or bf16 (bf16 and int4 experts). head_dim 64 or 128; n_heads / n_kv_heads in
 *   {1, 2, 4, 8}; d a multiple of 16 bytes of activations; d and n_heads * head_dim at most 12288;
 *   max_pos = KV-cache rows per layer. Allocates every layer's weights and caches on the handle's
 *   device. MOE_ERR_INVALID / MOE_ERR_OOM with the message in moe_decoder_last_error(NULL).
 * moe_decoder_set_layer: host pointers, copied: wq [n_heads*head_dim x d], wk and wv
 *   [n_kv_heads*head_dim x d], wo [d x n_heads*head_dim] (row-major, out x in), norm_in and
 *   norm_post [d], norm_q and norm_k [head_dim].
 * moe_decoder_set_cache: host K and V [n_kv_heads x n_pos x head_dim], copied into rows
 *   [0, n_pos) of the layer's cache, which then holds n_pos positions (n_pos in [0, max_pos]).
 * moe_decoder_step: x_in device [d] in the activation storage (the stream entering layer 0);
 *   x_out device fp32 [d] (the stream after the last layer); layer_log NULL or device fp32
 *   [n_layers x 4 x d]: per layer the stream entering it, W_o o, the MoE input as stored, and the
 *   MoE output as stored. Every layer's cache must hold the same number p of positions; the step
 *   writes row p and reads rows 0..p, then every layer holds p + 1. Returns after enqueueing on
 *   stream. MOE_ERR_NOT_REGISTERED if a layer's weights are missing, MOE_ERR_CAPACITY when p =
 *   max_pos, the MoE's status (its message copied) if a MoE layer fails, which empties the pool;
 *   a failed step leaves the positions unchanged. Not thread-safe per decoder.
 * moe_decoder_position: positions each layer's cache holds (-1 for NULL). */
typedef struct moe_decoder moe_decoder;
typedef struct {
  int32_t n_heads, n_kv_heads, head_dim;
  int32_t reserved; /* 0 */
  int64_t max_pos;
  double eps, rope_theta;
} moe_decoder_config;
moe_status moe_decoder_create(moe_handle* moe, const moe_decoder_config* cfg, moe_decoder** out);
moe_status moe_decoder_set_layer(moe_decoder* dec, int32_t layer, const void* wq, const void* wk, const void* wv,
                                 const void* wo, const void* norm_in, const void* norm_post, const void* norm_q,
                                 const void* norm_k);
moe_status moe_decoder_set_cache(moe_decoder* dec, int32_t layer, const void* k, const void* v, int64_t n_pos);
moe_status moe_decoder_step(moe_decoder* dec, const void* x_in, float* x_out, float* layer_log, void* stream);
int64_t moe_decoder_position(const moe_decoder* dec);
const char* moe_decoder_last_error(const moe_decoder* dec);
void moe_decoder_destroy(moe_decoder* dec);

/* ---- Residency planner ------------------------------------------------------------------------
 * The library's host slot table (the code the MOE_SCHEDULE_HOST_COPY_ENGINE schedule runs, and
 * the same rules the device schedule's kernel applies) driven by expert selections the caller
 * supplies. It touches no GPU and holds no weights. Use it to size a cap or compare policies on
 * a recorded routing sequence: it returns the hit / miss / eviction records a decode step would
 * produce (paper Sec. 3, Fig. 1: slot group, lookup table, selective load and evict).
 *
 * moe_planner_create: n_layers * n_experts global ids (gid = layer * n_experts + expert), a slot
 *   group of min(cap_slots, n_layers * n_experts) slots, all free; policy MOE_POLICY_LRU,
 *   MOE_POLICY_ROTARY or MOE_POLICY_GUIDED (rules as for moe_config.policy). MOE_ERR_INVALID for bad sizes (the
 *   message is moe_planner_last_error(NULL)); *out is NULL on failure.
 * moe_planner_preload: as moe_preload: free slots take absent ids in ascending order; those
 *   count as used before every step. *n_loaded (optional) = ids placed.
 * moe_planner_step: one layer-step. (step, layer) must increase from call to call (layer in
 *   [0, n_layers)) and orders the layer-steps for recency, as in a decode step. experts: the n expert ids (within
 *   the layer) the step uses; duplicates are merged, as the union of a batch's selections is.
 *   prefetch (LRU only, else MOE_ERR_INVALID): n_prefetch candidate ids admitted after the step,
 *   one reading of the paper's residency decisions that use information produced during
 *   execution (Sec. 3), e.g. the experts the router ranks right after its top k: ids that are
 *   absent take the lowest free slot, else the slot of the resident with the smallest
 *   (last use, gid) that is neither used by this step nor a candidate; when none is left the rest
 *   are dropped; an admitted id counts as used by this step. ranks: MOE_POLICY_GUIDED only (NULL
 *   otherwise), the rank in [0, n_experts] of each of the layer's n_experts experts in this step's
 *   routing (0 = highest logit; the best rank over a batch), applied before the lookup; a layer
 *   counts every expert at rank n_experts until its first step. recs (recs_cap >= n + n_prefetch)
 *   receives one record per distinct used id (ascending gid, kind 0 or 1) followed by one per
 *   admitted candidate (ascending, kind 2); *n_recs = records written. MOE_ERR_CAPACITY when a
 *   used id finds no slot (cap below the step's distinct ids): the records decided before it are
 *   written and the planner refuses further steps. Argument errors change nothing.
 * One planner is used by one host thread at a time. */
typedef struct moe_planner moe_planner;
moe_status moe_planner_create(int32_t n_layers, int32_t n_experts, int64_t cap_slots, int32_t policy,
                              moe_planner** out);
moe_status moe_planner_preload(moe_planner* p, int64_t* n_loaded);
moe_status moe_planner_step(moe_planner* p, int64_t step, int32_t layer, const int32_t* experts, int32_t n,
                            const int32_t* prefetch, int32_t n_prefetch, const int32_t* ranks, moe_trace_rec* recs,
                            int32_t recs_cap, int32_t* n_recs);
/* Message of the last failure on p (or of the last failed moe_planner_create if p is NULL). */
const char* moe_planner_last_error(const moe_planner* p);
/* NULL is a no-op. */
void moe_planner_destroy(moe_planner* p);

/* Paper: no counterpart (error reporting of this ABI).
 * Message of the last failure on h (or of the last failed moe_create if h is NULL). */
const char* moe_last_error(const moe_handle* h);

/* Paper: no counterpart (releases the slot group, the host tier and the work buffers).
 * Wait for outstanding work, free everything. NULL is a no-op. */
void moe_destroy(moe_handle* h);

#ifdef __cplusplus
}
#endif

#endif /* MOE_H_ */
