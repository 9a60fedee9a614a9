// C ABI of the capped-residency MoE decode library: handle, pinned host tier, slot pool,
// residency table (LRU with lower-id ties, or the rotary slot group), miss-copy pipeline and the
// per-layer schedules.
//
// Device schedule: one cooperative kernel per decode step runs every layer (fused.cu at batch 1,
// fused_batched.cu for batches, on tensor cores where the shape allows); the lookup table lives in
// device memory. This file sets up its state, launches it and reads back its error flag.
//
// Host-driven schedule of one layer (the routing result reaches the host through mapped
// pinned memory; the host owns the lookup table and issues the selective loads):
//   compute stream:  router(l) ............................ gateup(hits) [wait copy m] gateup(m) ... down+combine(l) router(l+1)
//   host:                      wait routing(l) -> LRU -> issue miss copies -> enqueue kernels
//   copy stream:                                 copy(m0) copy(m1) ...
// A slot is overwritten only by a copy issued after the host saw router(l) finish; router(l)
// runs after every kernel of layers < l on the compute stream, so no earlier reader of a
// victim slot can still be running, and experts needed by layer l are pinned for the step.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <chrono>
#include <cstdio>
#include <cstring>
#include <thread>
#include <string>
#include <utility>
#include <vector>

#include "fused.cuh"
#include "kernels.cuh"
#include "moe.h"
#include "moe_internal.h"
#include "slot_table.h"

namespace {

// NVTX range over a scope, optionally tagged with an integer (a layer): visible to nsys and to
// ncu --nvtx, a no-op when no tool is attached.
struct NvtxRange {
  explicit NvtxRange(const char* name, int tag = -1) {
    nvtxEventAttributes_t a{};
    a.version = NVTX_VERSION;
    a.size = NVTX_EVENT_ATTRIB_STRUCT_SIZE;
    a.messageType = NVTX_MESSAGE_TYPE_ASCII;
    a.message.ascii = name;
    if (tag >= 0) {
      a.payloadType = NVTX_PAYLOAD_TYPE_INT32;
      a.payload.iValue = tag;
    }
    nvtxRangePushEx(&a);
  }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

constexpr double kWaitTimeoutS = 20.0;
// CTAs of the fused kernel that stream missed experts: enough warps to keep the host link's
// bandwidth-delay product in flight when a layer-step misses only a few small (int4) experts,
// few enough not to flood it with outstanding requests when it misses several bf16 experts
// (measured on the 48-layer stacks: bf16 flat from 24 to 64 CTAs, int4 +8% at 64).
constexpr int kDefaultMissCtas = 64;
// The lookahead kernel keeps its miss CTAs streaming from one layer's misses to the next, so more of
// them pay (measured with 32 / 64 / 96 / 128 / 192 CTAs: int4 stack 470 / 551 / 582 / 531 / 445
// tok/s, bf16 stack 119 / 127 / 129 tok/s at 32 / 64 / 96).
constexpr int kDefaultMissCtasLookahead = 96;

thread_local std::string g_create_error;

enum {
  PC_ROUTER = 0, PC_GATEUP = 1, PC_DOWN = 2, PC_COPY = 3, PC_FUSED = 4,
  PC_PH_R = 5, PC_PH_S = 6, PC_PH_C = 7, PC_PH_D = 8, PC_PH_T = 9, PC_PH_E = 10, PC_PH_G = 11, PC_N = 12
};
const char* kPcName[PC_N] = {"router", "gateup", "down_combine", "miss_copy", "fused_step",
                             "fused_phase_router", "fused_phase_select", "fused_phase_gateup",
                             "fused_phase_down", "fused_phase_topk", "fused_phase_combine",
                             "fused_phase_gather"};

struct PendingTime {
  int cls;
  cudaEvent_t a, b;
  int64_t bytes;
};

}  // namespace

struct moe_handle {
  moe_config cfg{};
  moe::BlobLayout lay{};
  int64_t slot_stride = 0;
  int64_t n_gid = 0;
  int64_t cap = 0;
  int64_t asize = 0;         // activation element bytes
  int64_t router_eb = 0;     // router element bytes
  uint8_t* pool = nullptr;   // device slot pool
  bool own_pool = false;
  uint8_t* arena = nullptr;  // pinned host tier, one slot image per global expert id
  size_t arena_bytes = 0;
  std::vector<uint8_t> registered;
  std::vector<uint8_t> router_set;
  bool all_registered = false;
  uint8_t* routers = nullptr;  // device [L][E][d]
  moe::RouteOut* route = nullptr;      // mapped pinned (host view)
  moe::RouteOut* route_dev = nullptr;  // device view of the same memory
  float* u = nullptr;  // device [k][I]
  cudaStream_t copy_stream = nullptr;
  cudaStream_t host_stream = nullptr;
  std::vector<cudaEvent_t> copy_ev;
  cudaEvent_t layer_ev[2] = {nullptr, nullptr};  // host schedule with lookahead: layer l's last kernel done
  void* hid_dev = nullptr;
  void* out_dev = nullptr;
  // residency state of the host-driven schedule
  moe::SlotTable table;
  std::vector<int32_t> need_gids;
  std::vector<moe::SlotDecision> decisions;
  int64_t token_step = 0;
  int64_t route_seq = 0;
  std::vector<moe_trace_rec> trace;
  int64_t trace_dropped = 0;
  moe_stats stats{};
  std::vector<int32_t> last_idx;
  std::vector<float> last_gate;
  std::vector<float> last_z;      // host schedule, router-guided: [L][E] logits of the last step
  std::vector<int32_t> ranks;     // host schedule, router-guided: scratch [E]
  // profiling
  bool prof = false;
  std::vector<PendingTime> pending;
  std::vector<cudaEvent_t> ev_pool;
  double pc_ms[PC_N] = {};
  int64_t pc_launches[PC_N] = {};
  int64_t pc_bytes[PC_N] = {};
  unsigned long long* d_phase_ts = nullptr;   // [L*phases+1] per-phase timestamps of the last profiled step
  std::vector<unsigned long long> h_phase_ts;
  // device-driven schedule: lookup table, scratch and outputs in device memory
  bool dev_mode = false;
  bool batched = false;    // device schedule with max_batch > 1: the batched kernel
  bool batched_tc = false; // ... in its tensor-core variant
  CUtensorMap map_gu{}, map_d{}, map_x{}, map_u{};
  __nv_bfloat16* d_xg = nullptr;  // tensor-core variant: pairs' activations / u in plan order
  __nv_bfloat16* d_ug = nullptr;
  int fgrid = 0;
  int tg_max = 0;
  int touch_shift = 12;
  unsigned bar_epoch = 0;  // grid-barrier counter value at the start of the next fused launch
  bool lookahead_dev = false;  // device schedule with exact layer lookahead (k_fused_la) for whole steps
  int fgrid_la = 0;
  int la_group = 1;            // layers per worker barrier of the lookahead kernel
  int la_skew = 0;             // lookahead kernel: down rows of a group after the next group's gate/up rows
  unsigned wbar_epoch[2] = {0, 0};  // its worker arrival counters (by group parity) at the next launch
  const uint8_t* arena_dev = nullptr;
  // host time of the last decode-step launch (device schedule): after an idle gap the first step
  // re-reads one word per page of the host tier first (see decode_device)
  std::chrono::steady_clock::time_point last_launch{};
  bool launched = false;
  int32_t* d_slot_of = nullptr;
  unsigned long long* d_slot_key = nullptr;
  unsigned long long* d_cand = nullptr;  // batch-1 kernel: victim candidates [kMaxRanks + 1]
  int32_t* d_prior = nullptr;            // rotary policy: previous occupant per slot [cap]
  int32_t* d_prior_slot_of = nullptr;    // rotary policy: its inverse [n_gid]
  int32_t* d_rank = nullptr;             // router-guided policy: rank in the layer's latest routing [n_gid]
  int32_t* d_rank_best = nullptr;        // router-guided, batched: the layer-step's best rank [256]
  int32_t* d_hand = nullptr;             // rotary policy: the hand [1]
  int32_t* d_n_used = nullptr;
  int64_t* d_step = nullptr;
  float* d_z = nullptr;
  int32_t* d_plan = nullptr;  // batch 1: slot[k], gid[k], miss[k]; batched: n, nm, 5 x [E], pairs[Bmax*k]
  float* d_plan_gate = nullptr;  // batch 1: gate[k]; batched: gate per pair [Bmax*k]
  int32_t* d_sel_e = nullptr;    // batched: expert per pair [Bmax*k]
  float* d_y = nullptr;          // batched: W_d u per pair [Bmax*k][d]
  moe::TraceRec* d_trace = nullptr;
  unsigned long long* d_trace_n = nullptr;
  int32_t* d_route_idx = nullptr;
  float* d_route_gate = nullptr;
  unsigned long long* d_stats = nullptr;
  unsigned* d_bar = nullptr;  // barrier count, plan flag, then [2]: batched work-item counters or the
                              // lookahead kernel's worker arrival counters
  int* d_err = nullptr;
  int* h_err = nullptr;       // pinned copy of d_err after each step
  cudaEvent_t err_ev = nullptr;
  bool err_pending = false;
  int64_t steps_launched = 0;
  int fault = MOE_FAULT_NONE;  // armed by moe_inject_fault for the next decode step
  std::string err;
};

namespace {

moe_status fail(moe_handle* h, moe_status st, const std::string& msg) {
  if (h)
    h->err = msg;
  else
    g_create_error = msg;
  return st;
}

moe_status cuda_fail(moe_handle* h, cudaError_t e, const char* what) {
  return fail(h, MOE_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

#define MOE_CK(h, call)                                          \
  do {                                                           \
    cudaError_t e_ = (call);                                     \
    if (e_ != cudaSuccess) return cuda_fail((h), e_, #call);     \
  } while (0)

int64_t align_up(int64_t v, int64_t a) { return (v + a - 1) / a * a; }

// Returns an error message for an invalid configuration, or "" if cfg is usable.
std::string check_config(const moe_config* c) {
  if (!c) return "cfg is NULL";
  if (c->d <= 0 || c->n_experts <= 0 || c->top_k <= 0 || c->d_ff <= 0 || c->n_layers <= 0)
    return "d, n_experts, top_k, d_ff and n_layers must be positive";
  if (c->n_experts > 256) return "n_experts must be <= 256";
  if (c->top_k > moe::kMaxRanks || c->top_k > c->n_experts) return "top_k must be <= 16 and <= n_experts";
  if (c->max_batch < 1 || c->max_batch > moe::kMaxBatch) return "max_batch must be in [1, 64]";
  if (c->max_batch > 1 && c->schedule != MOE_SCHEDULE_DEVICE) return "max_batch above 1 needs the device schedule";
  if ((int64_t)c->n_layers * c->n_experts > 0x7fffffffLL) return "too many experts";
  if (c->wdtype == MOE_DTYPE_FP32) {
    if (c->adtype != MOE_DTYPE_FP32) return "fp32 weights need fp32 activations";
    if (c->d % 4 || c->d_ff % 4) return "fp32 needs d and d_ff multiples of 4";
    if (c->d > 2048) return "fp32 needs d <= 2048";
  } else if (c->wdtype == MOE_DTYPE_BF16) {
    if (c->adtype != MOE_DTYPE_BF16) return "bf16 weights need bf16 activations";
    if (c->d % 8 || c->d_ff % 8) return "bf16 needs d and d_ff multiples of 8";
    if (c->d > 4096) return "bf16 needs d <= 4096";
  } else if (c->wdtype == MOE_DTYPE_INT4_G128) {
    if (c->adtype != MOE_DTYPE_BF16) return "int4 weights need bf16 activations";
    if (c->d % 128 || c->d_ff % 128) return "int4 g128 needs d and d_ff multiples of 128";
    if (c->d > 16384) return "int4 needs d <= 16384";
  } else {
    return "unknown wdtype";
  }
  // down-projection chunks per lane (<= 8) and the u staging in shared memory
  const int64_t eb2 = c->wdtype == MOE_DTYPE_FP32 ? 8 : c->wdtype == MOE_DTYPE_BF16 ? 4 : 1;  // 2x bytes/elem
  if ((int64_t)c->d_ff * eb2 / 2 > 8 * 32 * 16) return "d_ff too large for the down-projection kernel";
  const int64_t ipad = align_up(c->d_ff, 32) + 4 * (align_up(c->d_ff, 32) / 32);
  if (c->max_batch == 1 && (int64_t)c->top_k * ipad * 4 > 200 * 1024)
    return "top_k * d_ff too large for shared-memory staging";
  if (c->renorm != 0 && c->renorm != 1) return "renorm must be 0 or 1";
  if (c->trace_capacity < 0) return "trace_capacity must be >= 0";
  if (c->schedule != MOE_SCHEDULE_DEVICE && c->schedule != MOE_SCHEDULE_HOST_COPY_ENGINE) return "unknown schedule";
  if (c->miss_ctas < 0) return "miss_ctas must be >= 0";
  if (c->batched_path != MOE_BATCHED_AUTO && c->batched_path != MOE_BATCHED_CUDA_CORES) return "unknown batched_path";
  if (c->policy != MOE_POLICY_LRU && c->policy != MOE_POLICY_ROTARY && c->policy != MOE_POLICY_GUIDED)
    return "unknown policy";
  if (c->policy == MOE_POLICY_GUIDED && (int64_t)c->n_layers * c->n_experts >= (1LL << moe::kGuidedGidBits))
    return "the router-guided policy needs n_layers * n_experts < 2^23";
  if (c->lookahead != 0 && c->lookahead != 1) return "lookahead must be 0 or 1";
  if (c->lookahead && c->schedule == MOE_SCHEDULE_DEVICE && (c->max_batch != 1 || c->policy != MOE_POLICY_LRU))
    return "lookahead in the device schedule needs max_batch 1 and the LRU policy";
  return "";
}

int64_t slots_for(const moe_config* c, int64_t stride) {
  int64_t cap = c->cap_slots > 0 ? c->cap_slots : (c->cap_bytes > 0 ? c->cap_bytes / stride : 0);
  const int64_t n_gid = (int64_t)c->n_layers * c->n_experts;
  return std::min(cap, n_gid);
}

void reset_device_state(moe_handle* h) {
  if (!h->dev_mode) return;
  cudaMemset(h->d_slot_of, 0xff, sizeof(int32_t) * h->n_gid);
  cudaMemset(h->d_slot_key, 0xff, sizeof(unsigned long long) * h->cap);
  cudaMemset(h->d_cand, 0, sizeof(unsigned long long) * (moe::kMaxRanks + 1));
  cudaMemset(h->d_prior, 0xff, sizeof(int32_t) * h->cap);
  cudaMemset(h->d_prior_slot_of, 0xff, sizeof(int32_t) * h->n_gid);
  {
    const std::vector<int32_t> unrouted((size_t)h->n_gid, h->cfg.n_experts);  // rank E: not routed yet
    cudaMemcpy(h->d_rank, unrouted.data(), sizeof(int32_t) * h->n_gid, cudaMemcpyHostToDevice);
  }
  cudaMemset(h->d_hand, 0, sizeof(int32_t));
  cudaMemset(h->d_n_used, 0, sizeof(int32_t));
  cudaMemset(h->d_step, 0, sizeof(int64_t));
  cudaMemset(h->d_trace_n, 0, sizeof(unsigned long long));
  cudaMemset(h->d_stats, 0, sizeof(unsigned long long) * moe::STAT_N);
  cudaMemset(h->d_bar, 0, sizeof(unsigned) * 4);
  h->bar_epoch = 0;
  h->wbar_epoch[0] = h->wbar_epoch[1] = 0;
  cudaMemset(h->d_err, 0, sizeof(int));
  cudaDeviceSynchronize();
  *h->h_err = 0;
  h->err_pending = false;
  h->steps_launched = 0;
  h->launched = false;  // the next step re-reads the host tier's pages first
}

void reset_state(moe_handle* h) {
  reset_device_state(h);
  h->table.reset();
  h->token_step = 0;
  h->trace.clear();
  h->trace_dropped = 0;
  h->stats = moe_stats{};
}

cudaEvent_t get_event(moe_handle* h) {
  if (!h->ev_pool.empty()) {
    cudaEvent_t e = h->ev_pool.back();
    h->ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Accumulate finished timing pairs (all pairs when `all`, else only those whose end event has
// completed) and recycle their events.
void harvest(moe_handle* h, bool all) {
  size_t keep = 0;
  for (size_t i = 0; i < h->pending.size(); i++) {
    PendingTime& p = h->pending[i];
    bool done = all ? (cudaEventSynchronize(p.b) == cudaSuccess) : (cudaEventQuery(p.b) == cudaSuccess);
    if (!done && !all) {
      h->pending[keep++] = p;
      continue;
    }
    float ms = 0.f;
    if (done && cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) {
      h->pc_ms[p.cls] += ms;
      h->pc_launches[p.cls] += 1;
      h->pc_bytes[p.cls] += p.bytes;
    }
    h->ev_pool.push_back(p.a);
    h->ev_pool.push_back(p.b);
  }
  h->pending.resize(keep);
  cudaGetLastError();
}

struct ProfScope {
  moe_handle* h;
  cudaStream_t s;
  int cls;
  int64_t bytes;
  cudaEvent_t a = nullptr;
  ProfScope(moe_handle* h_, cudaStream_t s_, int cls_, int64_t bytes_) : h(h_), s(s_), cls(cls_), bytes(bytes_) {
    if (h->prof) {
      a = get_event(h);
      if (a) cudaEventRecord(a, s);
    }
  }
  void done() {
    if (!a) return;
    cudaEvent_t b = get_event(h);
    if (!b) return;
    cudaEventRecord(b, s);
    h->pending.push_back(PendingTime{cls, a, b, bytes});
    a = nullptr;
  }
};

moe_status wait_route(moe_handle* h, int64_t seq, cudaStream_t s) {
  const auto t0 = std::chrono::steady_clock::now();
  uint64_t spins = 0;
  const volatile int64_t* p = &h->route->seq;
  for (;;) {
    if (__atomic_load_n((const int64_t*)p, __ATOMIC_ACQUIRE) == seq) return MOE_OK;
    if ((++spins & 4095) == 0) {
      cudaError_t e = cudaStreamQuery(s);
      if (e != cudaSuccess && e != cudaErrorNotReady) return cuda_fail(h, e, "device fault while waiting for routing");
      const double dt = std::chrono::duration<double>(std::chrono::steady_clock::now() - t0).count();
      if (dt > kWaitTimeoutS) return fail(h, MOE_ERR_TIMEOUT, "timed out waiting for the routing result");
    }
  }
}

moe_status launch_router(moe_handle* h, int32_t layer, const void* hidden_l, cudaStream_t s) {
  moe::RouterArgs a{};
  a.w = h->routers + (int64_t)layer * h->cfg.n_experts * h->cfg.d * h->router_eb;
  a.h = hidden_l;
  a.E = h->cfg.n_experts;
  a.d = h->cfg.d;
  a.k = h->cfg.top_k;
  a.renorm = h->cfg.renorm;
  a.wdtype = h->cfg.wdtype == MOE_DTYPE_FP32 ? moe::WD_FP32 : moe::WD_BF16;
  a.out = h->route_dev;
  a.seq = ++h->route_seq;
  a.want_z = h->cfg.policy == MOE_POLICY_GUIDED;
  ProfScope ps(h, s, PC_ROUTER, (int64_t)a.E * a.d * h->router_eb + (int64_t)a.d * h->asize);
  cudaError_t e = moe::launch_router(a, s);
  ps.done();
  if (e != cudaSuccess) return cuda_fail(h, e, "router launch");
  return MOE_OK;
}

struct Need {
  int32_t gid;
  int32_t slot;
  bool miss;
  int32_t evicted;  // global id the miss evicted, -1 if none
};

// One layer-step of the lookup table (rules in slot_table.h; needs in ascending gid). Fills each
// need's slot and miss flag, the stats and the trace.
moe_status residency_step(moe_handle* h, int32_t layer, std::vector<Need>& needs, int64_t clock) {
  const int32_t E = h->cfg.n_experts;
  h->need_gids.clear();
  for (auto& n : needs) h->need_gids.push_back(n.gid);
  h->decisions.clear();
  const bool ok = h->table.step(h->need_gids.data(), (int32_t)h->need_gids.size(), clock, h->decisions);
  for (size_t i = 0; i < h->decisions.size(); i++) {
    const moe::SlotDecision& d = h->decisions[i];
    Need& n = needs[i];
    n.slot = d.slot;
    n.miss = d.kind == moe::SLOT_MISS;
    n.evicted = d.evicted;
    if (n.miss) {
      h->stats.misses++;
      h->stats.miss_bytes += h->lay.total;
      if (d.evicted >= 0) h->stats.evictions++;
    } else {
      h->stats.hits++;
    }
    if (h->cfg.trace_capacity > 0) {
      if ((int64_t)h->trace.size() < h->cfg.trace_capacity)
        h->trace.push_back(moe_trace_rec{(int32_t)h->token_step, layer, d.gid - layer * E, d.kind, d.slot, d.evicted});
      else
        h->trace_dropped++;
    }
  }
  if (!ok) return fail(h, MOE_ERR_CAPACITY, "no slot available (cap below the layer-step's working set)");
  return MOE_OK;
}

moe_status decode_impl(moe_handle* h, const void* hidden, void* out, cudaStream_t s) {
  const moe_config& c = h->cfg;
  const int32_t L = c.n_layers, E = c.n_experts, k = c.top_k;
  const int64_t act_row = (int64_t)c.d * h->asize;
  const int64_t gu_bytes = h->lay.d_off;              // GU rows + GU scales
  const int64_t dn_bytes = h->lay.total - h->lay.d_off;  // D rows + D scales
  if (h->prof) harvest(h, false);
  h->last_idx.assign((size_t)L * k, -1);
  h->last_gate.assign((size_t)L * k, 0.f);
  if (c.policy == MOE_POLICY_GUIDED) h->last_z.assign((size_t)L * E, 0.f);
  moe_status st = launch_router(h, 0, hidden, s);
  if (st != MOE_OK) return st;
  std::vector<Need> needs;
  std::vector<int32_t> rank_gid(k);
  std::vector<int32_t> prev_needed;  // lookahead: the global ids layer l - 1 reads
  for (int32_t l = 0; l < L; l++) {
    const void* hid_l = (const uint8_t*)hidden + (int64_t)l * act_row;
    NvtxRange layer_range("layer", l);
    {
      NvtxRange r("wait for routing", l);
      st = wait_route(h, h->route_seq, s);
    }
    if (st != MOE_OK) return st;
    if (h->prof) harvest(h, false);
    // routing result of layer l
    needs.clear();
    const volatile int32_t* ridx = h->route->idx;
    const volatile float* rgate = h->route->gate;
    for (int32_t r = 0; r < k; r++) {
      const int32_t e = ridx[r];
      if (e < 0 || e >= E) return fail(h, MOE_ERR_INVALID, "router produced an invalid expert id (non-finite logits?)");
      h->last_idx[(size_t)l * k + r] = e;
      h->last_gate[(size_t)l * k + r] = rgate[r];
      rank_gid[r] = l * E + e;
      needs.push_back(Need{l * E + e, -1, false, -1});
    }
    std::sort(needs.begin(), needs.end(), [](const Need& a, const Need& b) { return a.gid < b.gid; });
    if (c.policy == MOE_POLICY_GUIDED) {
      // the layer's ranks from this routing: the logits that beat each expert's, ties to the
      // lower id (the router's own order)
      float* zl = h->last_z.data() + (size_t)l * E;
      const volatile float* rz = h->route->z;
      for (int32_t e = 0; e < E; e++) zl[e] = rz[e];
      h->ranks.resize(E);
      for (int32_t e = 0; e < E; e++) {
        int32_t r = 0;
        for (int32_t j = 0; j < E; j++) r += (zl[j] > zl[e] || (zl[j] == zl[e] && j < e)) ? 1 : 0;
        h->ranks[e] = r;
      }
      h->table.set_ranks(l, h->ranks.data());
    }
    for (size_t i = 1; i < needs.size(); i++)
      if (needs[i].gid == needs[i - 1].gid) return fail(h, MOE_ERR_INVALID, "router produced duplicate expert ids");
    // Lookahead: layer l's routing is in host arrays now, so layer l + 1's router may overwrite the
    // routing buffer. Launched here, it runs on the GPU before layer l's kernels enqueued below,
    // and the next iteration issues layer l + 1's miss copies while layer l computes.
    if (c.lookahead && l + 1 < L) {
      st = launch_router(h, l + 1, (const uint8_t*)hidden + (int64_t)(l + 1) * act_row, s);
      if (st != MOE_OK) return st;
    }
    const int64_t clock = h->token_step * L + l + 1;  // 0 is older than every step (preloaded experts)
    {
      NvtxRange r("slot lookup", l);
      st = residency_step(h, l, needs, clock);
    }
    if (st != MOE_OK) return st;
    h->stats.layer_steps++;
    // selective loads: misses in ascending gid on the copy stream
    int n_miss = 0;
    bool waited_prev = false;
    for (auto& n : needs) {
      if (!n.miss) continue;
      // Lookahead: layer l - 1's kernels may still be running. A victim they read is overwritten
      // only after its last kernel (every layer before it has finished: layer l's router ran
      // after it). With cap >= 2 x a layer-step's experts an LRU victim is never such an expert.
      if (c.lookahead && !waited_prev && n.evicted >= 0 &&
          std::find(prev_needed.begin(), prev_needed.end(), n.evicted) != prev_needed.end()) {
        MOE_CK(h, cudaStreamWaitEvent(h->copy_stream, h->layer_ev[(l - 1) & 1], 0));
        waited_prev = true;
      }
      ProfScope ps(h, h->copy_stream, PC_COPY, h->lay.total);
      if (h->fault == MOE_FAULT_COPY_ERROR) {  // an armed copy fault: this copy "fails"
        h->fault = MOE_FAULT_NONE;
        return cuda_fail(h, cudaErrorInvalidValue, "miss copy (injected fault)");
      }
      MOE_CK(h, cudaMemcpyAsync(h->pool + (int64_t)n.slot * h->slot_stride, h->arena + (int64_t)n.gid * h->slot_stride,
                                h->lay.total, cudaMemcpyHostToDevice, h->copy_stream));
      ps.done();
      MOE_CK(h, cudaEventRecord(h->copy_ev[n_miss], h->copy_stream));
      n_miss++;
    }
    auto slot_ptr = [&](int32_t gid) { return h->pool + (int64_t)h->table.slot_of(gid) * h->slot_stride; };
    // gate-up on the hits
    moe::GateUpArgs ga{};
    ga.d = c.d;
    ga.I = c.d_ff;
    ga.lay = h->lay;
    ga.x = hid_l;
    ga.n_tasks = 0;
    for (int32_t r = 0; r < k; r++) {
      const Need* n = nullptr;
      for (auto& x : needs)
        if (x.gid == rank_gid[r]) n = &x;
      if (n->miss) continue;
      ga.blob[ga.n_tasks] = slot_ptr(rank_gid[r]);
      ga.u[ga.n_tasks] = h->u + (int64_t)r * c.d_ff;
      ga.n_tasks++;
    }
    if (ga.n_tasks > 0) {
      ProfScope ps(h, s, PC_GATEUP, (int64_t)ga.n_tasks * gu_bytes);
      cudaError_t e = moe::launch_gateup(ga, c.wdtype, s);
      ps.done();
      if (e != cudaSuccess) return cuda_fail(h, e, "gate-up launch");
    }
    // gate-up on each miss once its copy has landed
    int m = 0;
    for (auto& n : needs) {
      if (!n.miss) continue;
      MOE_CK(h, cudaStreamWaitEvent(s, h->copy_ev[m], 0));
      m++;
      ga.n_tasks = 0;
      for (int32_t r = 0; r < k; r++) {
        if (rank_gid[r] != n.gid) continue;
        ga.blob[ga.n_tasks] = slot_ptr(n.gid);
        ga.u[ga.n_tasks] = h->u + (int64_t)r * c.d_ff;
        ga.n_tasks++;
      }
      ProfScope ps(h, s, PC_GATEUP, (int64_t)ga.n_tasks * gu_bytes);
      cudaError_t e = moe::launch_gateup(ga, c.wdtype, s);
      ps.done();
      if (e != cudaSuccess) return cuda_fail(h, e, "gate-up launch");
    }
    // down projection + rank-ordered combine
    moe::DownArgs da{};
    da.k = k;
    da.d = c.d;
    da.I = c.d_ff;
    da.lay = h->lay;
    for (int32_t r = 0; r < k; r++) {
      da.blob[r] = slot_ptr(rank_gid[r]);
      da.gate[r] = h->last_gate[(size_t)l * k + r];
    }
    da.u = h->u;
    da.out = (uint8_t*)out + (int64_t)l * act_row;
    {
      ProfScope ps(h, s, PC_DOWN, (int64_t)k * dn_bytes);
      cudaError_t e = moe::launch_down_combine(da, c.wdtype, s);
      ps.done();
      if (e != cudaSuccess) return cuda_fail(h, e, "down/combine launch");
    }
    if (c.lookahead) {
      MOE_CK(h, cudaEventRecord(h->layer_ev[l & 1], s));
      prev_needed.clear();
      for (auto& n : needs) prev_needed.push_back(n.gid);
    } else if (l + 1 < L) {
      st = launch_router(h, l + 1, (const uint8_t*)hidden + (int64_t)(l + 1) * act_row, s);
      if (st != MOE_OK) return st;
    }
  }
  h->token_step++;
  h->stats.steps++;
  return MOE_OK;
}

// The host tier: page-locked, device-mapped host memory from the CUDA allocator. Warps of the
// decode kernels read missed experts from it directly over NVLink-C2C. Memory allocated this way
// sustained the link's full rate (~200 GB/s) for SM reads; anonymous memory page-locked with
// cudaHostRegister read at half that, varying from run to run.
moe_status alloc_arena(moe_handle* h) {
  const size_t bytes = (size_t)(h->n_gid * h->slot_stride);
  void* p = nullptr;
  if (cudaHostAlloc(&p, bytes, cudaHostAllocMapped) != cudaSuccess) {
    cudaGetLastError();
    return fail(h, MOE_ERR_OOM, "page-locked host arena allocation failed (" + std::to_string(bytes >> 20) + " MiB)");
  }
  h->arena = (uint8_t*)p;
  h->arena_bytes = bytes;
  return MOE_OK;
}

// Device-driven schedule: report a failure flagged by an earlier fused step. With sync, waits for
// all work and reads the live flag; otherwise reads the copy taken after the last completed step.
// A flagged failure empties the pool and clears the flag.
moe_status check_device_error(moe_handle* h, bool sync) {
  if (!h->dev_mode) return MOE_OK;
  int e = 0;
  if (sync) {
    cudaError_t ce = cudaDeviceSynchronize();
    if (ce != cudaSuccess) return cuda_fail(h, ce, "decode step");
    ce = cudaMemcpy(&e, h->d_err, sizeof(int), cudaMemcpyDeviceToHost);
    if (ce != cudaSuccess) return cuda_fail(h, ce, "reading the device error flag");
  } else if (h->err_pending && cudaEventQuery(h->err_ev) == cudaSuccess) {
    e = *(volatile int*)h->h_err;
  }
  cudaGetLastError();
  if (e == 0) return MOE_OK;
  std::string msg = "decode step failed on the device:";
  if (e & moe::FERR_BARRIER_TIMEOUT) msg += " a grid barrier timed out;";
  if (e & moe::FERR_BAD_ROUTE) msg += " the router produced an invalid expert id (non-finite logits?);";
  if (e & moe::FERR_NO_VICTIM) msg += " no evictable slot;";
  if (e & moe::FERR_PIPE_TIMEOUT) msg += " a wait for copies into shared memory timed out;";
  msg += " the pool was emptied";
  reset_state(h);
  return fail(h, (e & moe::FERR_FATAL) ? MOE_ERR_TIMEOUT : MOE_ERR_CUDA, msg);
}

// Per-phase durations of the last profiled step from the kernel's global-timer stamps.
moe_status harvest_phases(moe_handle* h, const unsigned long long* d_ts, int nph, const int* cls, cudaStream_t s) {
  const int L = h->cfg.n_layers;
  h->h_phase_ts.resize((size_t)nph * L + 1);
  MOE_CK(h, cudaMemcpyAsync(h->h_phase_ts.data(), d_ts, sizeof(unsigned long long) * (nph * L + 1),
                            cudaMemcpyDeviceToHost, s));
  MOE_CK(h, cudaStreamSynchronize(s));
  unsigned long long prev = h->h_phase_ts[(size_t)nph * L];
  for (int l = 0; l < L; l++)
    for (int p = 0; p < nph; p++) {
      const unsigned long long t = h->h_phase_ts[(size_t)nph * l + p];
      h->pc_ms[cls[p]] += (double)(t - prev) * 1e-6;
      h->pc_launches[cls[p]] += 1;
      prev = t;
    }
  return MOE_OK;
}

unsigned long long* phase_buffer(moe_handle* h) {
  if (!h->prof) return nullptr;
  if (!h->d_phase_ts &&
      cudaMalloc(&h->d_phase_ts, sizeof(unsigned long long) * (moe::kBatchedTcPhases * h->cfg.n_layers + 1)) !=
          cudaSuccess) {
    h->d_phase_ts = nullptr;
    cudaGetLastError();
  }
  return h->d_phase_ts;
}

// An armed barrier fault: the step's grid barriers wait for an arrival count that no launch
// reaches, with a 0.2 s limit, so every CTA's bounded wait runs out and the step reports
// MOE_ERR_TIMEOUT (the kernels exit normally; nothing waits without a limit).
void arm_barrier_fault(moe_handle* h, unsigned& bar_base, unsigned long long& timeout_ns) {
  if (h->fault != MOE_FAULT_BARRIER_TIMEOUT) return;
  h->fault = MOE_FAULT_NONE;
  bar_base += 0x40000000u;
  timeout_ns = 200000000ull;
}

moe_status decode_batched(moe_handle* h, const void* hidden, void* out, int32_t batch, cudaStream_t s) {
  const moe_config& c = h->cfg;
  const int k = c.top_k, E = c.n_experts;
  moe::BatchArgs a{};
  a.L = c.n_layers;
  a.E = E;
  a.k = k;
  a.d = c.d;
  a.I = c.d_ff;
  a.renorm = c.renorm;
  a.wdtype = c.wdtype;
  a.B = batch;
  a.Bmax = c.max_batch;
  a.lay = h->lay;
  a.slot_stride = h->slot_stride;
  a.cap = h->cap;
  a.n_gid = h->n_gid;
  a.routers = h->routers;
  a.hidden = hidden;
  a.out = out;
  a.pool = h->pool;
  a.arena = h->arena_dev;
  a.slot_of = h->d_slot_of;
  a.slot_key = h->d_slot_key;
  a.n_used = h->d_n_used;
  a.step = h->d_step;
  a.z = h->d_z;
  a.sel_e = h->d_sel_e;
  a.sel_g = h->d_plan_gate;
  a.plan_n = h->d_plan;
  a.plan_slot = h->d_plan + 2;
  a.plan_gid = h->d_plan + 2 + E;
  a.plan_miss = h->d_plan + 2 + 2 * E;
  a.plan_off = h->d_plan + 2 + 3 * E;
  a.plan_cnt = h->d_plan + 2 + 4 * E;
  a.plan_tok = h->d_plan + 2 + 5 * E;
  a.u = h->u;
  a.y = h->d_y;
  a.trace = h->d_trace;
  a.trace_cap = c.trace_capacity;
  a.trace_n = h->d_trace_n;
  a.route_idx = h->d_route_idx;
  a.route_gate = h->d_route_gate;
  a.stats = h->d_stats;
  a.bar_count = h->d_bar;
  a.bar_base = h->bar_epoch;
  a.err = h->d_err;
  a.barrier_timeout_ns = 2000000000ull;
  arm_barrier_fault(h, a.bar_base, a.barrier_timeout_ns);
  a.phase_ts = phase_buffer(h);
  a.work = h->d_bar + 2;
  a.touch_shift = h->touch_shift;
  a.tg_max = h->tg_max;
  a.router_tb = moe::batched_router_tb(c.wdtype, c.d, c.d_ff, h->batched_tc);
  a.policy = c.policy;
  a.rank = h->d_rank;
  a.rank_best = h->d_rank_best;
  a.prior = h->d_prior;
  a.prior_slot_of = h->d_prior_slot_of;
  a.hand = h->d_hand;
  a.map_gu = h->map_gu;
  a.map_d = h->map_d;
  a.map_x = h->map_x;
  a.map_u = h->map_u;
  a.xg = h->d_xg;
  a.ug = h->d_ug;
  {
    ProfScope ps(h, s, PC_FUSED, (int64_t)c.n_layers * (int64_t)E * c.d * h->router_eb);
    cudaError_t e = h->batched_tc ? moe::launch_fused_batched_tc(a, h->fgrid, s) : moe::launch_fused_batched(a, h->fgrid, s);
    ps.done();
    if (e != cudaSuccess) return cuda_fail(h, e, "batched decode step launch");
  }
  MOE_CK(h, cudaMemcpyAsync(h->h_err, h->d_err, sizeof(int), cudaMemcpyDeviceToHost, s));
  MOE_CK(h, cudaEventRecord(h->err_ev, s));
  h->err_pending = true;
  h->steps_launched++;
  // every CTA arrives at each phase's barrier once per layer
  const int nph = h->batched_tc ? moe::kBatchedTcPhases : moe::kBatchedPhases;
  h->bar_epoch += (unsigned)nph * (unsigned)c.n_layers * (unsigned)h->fgrid;
  if (a.phase_ts) {
    static const int cls[moe::kBatchedPhases] = {PC_PH_R, PC_PH_T, PC_PH_S, PC_PH_C, PC_PH_D, PC_PH_E};
    static const int cls_tc[moe::kBatchedTcPhases] = {PC_PH_R, PC_PH_T, PC_PH_S, PC_PH_G, PC_PH_C, PC_PH_D, PC_PH_E};
    return harvest_phases(h, a.phase_ts, nph, h->batched_tc ? cls_tc : cls, s);
  }
  return MOE_OK;
}

// Layers [l0, l1) of a batch-1 decode step in one launch of the fused kernel; the launch that
// reaches the last layer completes the step. Per-phase profiling covers whole-step launches only.
moe_status decode_device_layers(moe_handle* h, const void* hidden, void* out, int32_t l0, int32_t l1,
                                cudaStream_t s) {
  const moe_config& c = h->cfg;
  const int k = c.top_k;
  const bool whole = l0 == 0 && l1 == c.n_layers;
  moe::FusedArgs a{};
  a.L = c.n_layers;
  a.l_begin = l0;
  a.l_end = l1;
  a.E = c.n_experts;
  a.k = k;
  a.d = c.d;
  a.I = c.d_ff;
  a.renorm = c.renorm;
  a.wdtype = c.wdtype;
  a.lay = h->lay;
  a.slot_stride = h->slot_stride;
  a.cap = h->cap;
  a.routers = h->routers;
  a.hidden = hidden;
  a.out = out;
  a.pool = h->pool;
  a.arena = h->arena_dev;
  a.slot_of = h->d_slot_of;
  a.slot_key = h->d_slot_key;
  a.cand = h->d_cand;
  a.policy = c.policy;
  a.may_evict = h->cap < h->n_gid && c.policy != MOE_POLICY_ROTARY;
  a.rank = h->d_rank;
  a.prior = h->d_prior;
  a.prior_slot_of = h->d_prior_slot_of;
  a.hand = h->d_hand;
  a.plan_flag = h->d_bar + 1;  // cleared with the barrier counter
  a.n_used = h->d_n_used;
  a.step = h->d_step;
  a.z = h->d_z;
  a.plan_slot = h->d_plan;
  a.plan_gid = h->d_plan + k;
  a.plan_miss = h->d_plan + 2 * k;
  a.plan_gate = h->d_plan_gate;
  a.u = h->u;
  a.trace = h->d_trace;
  a.trace_cap = c.trace_capacity;
  a.trace_n = h->d_trace_n;
  a.route_idx = h->d_route_idx;
  a.route_gate = h->d_route_gate;
  a.stats = h->d_stats;
  a.bar_count = h->d_bar;
  a.bar_base = h->bar_epoch;
  a.err = h->d_err;
  a.barrier_timeout_ns = 2000000000ull;
  arm_barrier_fault(h, a.bar_base, a.barrier_timeout_ns);
  a.miss_ctas =
      c.miss_ctas > 0 ? c.miss_ctas : (whole && h->lookahead_dev ? kDefaultMissCtasLookahead : kDefaultMissCtas);
  a.touch_shift = h->touch_shift;
  // whole steps of a lookahead handle: every layer's plan at plan[l][k], one grid barrier per launch
  const bool la = whole && h->lookahead_dev;
  if (la) {
    const int64_t Lk = (int64_t)c.n_layers * k;
    a.plan_gid = h->d_plan + Lk;
    a.plan_miss = h->d_plan + 2 * Lk;
    a.wbar_count = h->d_bar + 2;  // [2], free at batch 1
    a.wbar_base[0] = h->wbar_epoch[0];
    a.wbar_base[1] = h->wbar_epoch[1];
    a.la_group = h->la_group;
    a.la_skew = h->la_skew;
    a.may_evict = a.may_evict && c.policy == MOE_POLICY_LRU;
  }
  a.phase_ts = whole && !la ? phase_buffer(h) : nullptr;
  {
    ProfScope ps(h, s, PC_FUSED,
                 (int64_t)(l1 - l0) * (k * h->lay.total + (int64_t)c.n_experts * c.d * h->router_eb));
    cudaError_t e = la ? moe::launch_fused_la(a, h->fgrid_la, s) : moe::launch_fused(a, h->fgrid, s);
    ps.done();
    if (e != cudaSuccess) return cuda_fail(h, e, "fused decode step launch");
  }
  MOE_CK(h, cudaMemcpyAsync(h->h_err, h->d_err, sizeof(int), cudaMemcpyDeviceToHost, s));
  MOE_CK(h, cudaEventRecord(h->err_ev, s));
  h->err_pending = true;
  if (l1 == c.n_layers) h->steps_launched++;
  if (la) {
    h->bar_epoch += (unsigned)h->fgrid_la;  // one grid barrier (after the router phase)
    const unsigned groups = (unsigned)((c.n_layers + h->la_group - 1) / h->la_group);
    // every worker arrives once per layer group, on the counter of the group's parity
    h->wbar_epoch[0] += ((groups + 1) / 2) * (unsigned)(h->fgrid_la - 1);
    h->wbar_epoch[1] += (groups / 2) * (unsigned)(h->fgrid_la - 1);
  } else {
    h->bar_epoch += 3u * (unsigned)(l1 - l0) * (unsigned)h->fgrid;  // every CTA arrives at 3 barriers per layer
  }
  if (a.phase_ts) {
    // phase durations of this step (the copy waits for the step; profiling runs are not timed for overlap)
    static const int cls[4] = {PC_PH_R, PC_PH_S, PC_PH_C, PC_PH_D};
    return harvest_phases(h, a.phase_ts, 4, cls, s);
  }
  return MOE_OK;
}

moe_status check_registered(moe_handle* h) {
  if (h->all_registered) return MOE_OK;
  for (int32_t l = 0; l < h->cfg.n_layers; l++)
    if (!h->router_set[l]) return fail(h, MOE_ERR_NOT_REGISTERED, "router of layer " + std::to_string(l) + " not set");
  for (int64_t g = 0; g < h->n_gid; g++)
    if (!h->registered[g])
      return fail(h, MOE_ERR_NOT_REGISTERED, "expert " + std::to_string(g % h->cfg.n_experts) + " of layer " +
                                                 std::to_string(g / h->cfg.n_experts) + " not registered");
  h->all_registered = true;
  return MOE_OK;
}

// The pool contents are unknown after a failed step: wait for the streams, empty the pool.
void recover_after_failure(moe_handle* h, cudaStream_t s) {
  std::string keep = h->err;
  cudaStreamSynchronize(s);
  cudaStreamSynchronize(h->copy_stream);
  cudaGetLastError();
  reset_state(h);
  h->err = keep;
}

// After the host link has been idle for a while the SMs' reads of the host tier run 2-3x slower
// and recover only over ~1 s of streaming. Measured on GB300 with the 48-layer bf16 stack (58 GB
// tier): after 20 s idle (or right after the tier is built) the first 10 tokens took 23-28 ms each
// against 8.5-9 ms back to back, recovering over ~100 tokens (~0.7 s lost in all); after a 2 s gap
// the loss was ~20 ms; copy-engine traffic in the gap made no difference. One read per 4 KB page
// of the whole tier from all SMs at once before the first step after a gap of kIdleRewarm or more
// pays about the same once (0.5-0.7 s cold for 58 GB) and leaves the following steps at the loaded
// rate. Shorter gaps are left to recover by themselves (the pass costs ~50 ms even when warm).
constexpr std::chrono::milliseconds kIdleRewarm{2000};

// Enqueues the re-read pass on s before a step that follows an idle gap (device schedule).
moe_status rewarm_if_idle(moe_handle* h, cudaStream_t s) {
  const auto now = std::chrono::steady_clock::now();
  if (h->cap < h->n_gid && (!h->launched || now - h->last_launch >= kIdleRewarm)) {
    NvtxRange range("re-read the host tier's pages after an idle gap");
    MOE_CK(h, moe::launch_touch_pages(h->arena_dev, (int64_t)h->arena_bytes, 12, s));
  }
  h->last_launch = now;
  h->launched = true;
  return MOE_OK;
}

moe_status decode_device(moe_handle* h, const void* hidden, void* out, int32_t batch, cudaStream_t s) {
  moe_status st = check_device_error(h, false);
  if (st != MOE_OK) return st;
  st = rewarm_if_idle(h, s);
  if (st != MOE_OK) return st;
  if (h->batched) return decode_batched(h, hidden, out, batch, s);
  return decode_device_layers(h, hidden, out, 0, h->cfg.n_layers, s);
}

// The driver's tensor-map encoder, looked up once per process (thread-safe static initialisation).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    PFN_cuTensorMapEncodeTiled_v12000 f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f = (PFN_cuTensorMapEncodeTiled_v12000)p;
    cudaGetLastError();
    return f;
  }();
  return fn;
}

// bf16 tensor map with the 128-byte swizzle; dims[0] is the contiguous (K) dimension.
bool encode_map(CUtensorMap* m, void* base, cuuint32_t rank, const cuuint64_t* dims, const cuuint64_t* strides,
                const cuuint32_t* box) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, base, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Buffers and TMA maps of the tensor-core batched kernel: the weights in the slot pool, and the
// pairs' activations / u vectors in plan order (rows padded to a multiple of 16, zeroed).
moe_status make_tc_maps(moe_handle* h) {
  const moe_config& c = h->cfg;
  const int64_t rows = std::max<int64_t>(16, align_up((int64_t)c.max_batch * c.top_k, 16));
  if (cudaMalloc(&h->d_xg, rows * c.d * 2) != cudaSuccess || cudaMalloc(&h->d_ug, rows * c.d_ff * 2) != cudaSuccess)
    return fail(h, MOE_ERR_OOM, "tensor-core staging allocation failed");
  if (cudaMemset(h->d_xg, 0, rows * c.d * 2) != cudaSuccess || cudaMemset(h->d_ug, 0, rows * c.d_ff * 2) != cudaSuccess)
    return fail(h, MOE_ERR_CUDA, "tensor-core staging memset failed");
  const cuuint64_t dgu[3] = {(cuuint64_t)c.d, (cuuint64_t)(2 * c.d_ff), (cuuint64_t)h->cap};
  const cuuint64_t sgu[2] = {(cuuint64_t)c.d * 2, (cuuint64_t)h->slot_stride};
  const cuuint64_t dd[3] = {(cuuint64_t)c.d_ff, (cuuint64_t)c.d, (cuuint64_t)h->cap};
  const cuuint64_t sd[2] = {(cuuint64_t)c.d_ff * 2, (cuuint64_t)h->slot_stride};
  const cuuint32_t box_w[3] = {64, 128, 1};
  const cuuint64_t dx[2] = {(cuuint64_t)c.d, (cuuint64_t)rows};
  const cuuint64_t sx[1] = {(cuuint64_t)c.d * 2};
  const cuuint64_t du[2] = {(cuuint64_t)c.d_ff, (cuuint64_t)rows};
  const cuuint64_t su[1] = {(cuuint64_t)c.d_ff * 2};
  const cuuint32_t box_p[2] = {64, 16};
  if (!encode_map(&h->map_gu, h->pool, 3, dgu, sgu, box_w) ||
      !encode_map(&h->map_d, h->pool + h->lay.d_off, 3, dd, sd, box_w) ||
      !encode_map(&h->map_x, h->d_xg, 2, dx, sx, box_p) || !encode_map(&h->map_u, h->d_ug, 2, du, su, box_p))
    return fail(h, MOE_ERR_CUDA, "TMA tensor map encoding failed");
  return MOE_OK;
}

void free_all(moe_handle* h) {
  if (!h) return;
  cudaDeviceSynchronize();
  harvest(h, true);
  for (auto e : h->ev_pool) cudaEventDestroy(e);
  for (auto e : h->copy_ev) cudaEventDestroy(e);
  for (auto e : h->layer_ev)
    if (e) cudaEventDestroy(e);
  if (h->copy_stream) cudaStreamDestroy(h->copy_stream);
  if (h->host_stream) cudaStreamDestroy(h->host_stream);
  if (h->own_pool && h->pool) cudaFree(h->pool);
  if (h->arena) cudaFreeHost(h->arena);
  if (h->routers) cudaFree(h->routers);
  if (h->route) cudaFreeHost(h->route);
  if (h->u) cudaFree(h->u);
  for (void* p : {(void*)h->d_slot_of, (void*)h->d_slot_key, (void*)h->d_cand, (void*)h->d_prior,
                  (void*)h->d_prior_slot_of, (void*)h->d_rank, (void*)h->d_rank_best, (void*)h->d_hand,
                  (void*)h->d_n_used,
                  (void*)h->d_step, (void*)h->d_z, (void*)h->d_plan, (void*)h->d_plan_gate, (void*)h->d_trace,
                  (void*)h->d_trace_n, (void*)h->d_route_idx, (void*)h->d_route_gate, (void*)h->d_stats,
                  (void*)h->d_bar, (void*)h->d_err, (void*)h->d_phase_ts, (void*)h->d_sel_e, (void*)h->d_y,
                  (void*)h->d_xg, (void*)h->d_ug})
    if (p) cudaFree(p);
  if (h->h_err) cudaFreeHost(h->h_err);
  if (h->err_ev) cudaEventDestroy(h->err_ev);
  if (h->hid_dev) cudaFree(h->hid_dev);
  if (h->out_dev) cudaFree(h->out_dev);
  cudaGetLastError();
  delete h;
}

}  // namespace

extern "C" {

int64_t moe_expert_bytes(const moe_config* cfg) {
  if (!check_config(cfg).empty()) return -1;
  return moe::make_layout(cfg->wdtype, cfg->d, cfg->d_ff).total;
}

int64_t moe_pool_bytes(const moe_config* cfg) {
  if (!check_config(cfg).empty()) return -1;
  const int64_t stride = align_up(moe::make_layout(cfg->wdtype, cfg->d, cfg->d_ff).total, 256);
  return slots_for(cfg, stride) * stride;
}

moe_status moe_create(const moe_config* cfg, moe_handle** out) {
  if (!out) return fail(nullptr, MOE_ERR_INVALID, "out is NULL");
  *out = nullptr;
  std::string why = check_config(cfg);
  if (!why.empty()) return fail(nullptr, MOE_ERR_INVALID, why);
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || cfg->device < 0 || cfg->device >= ndev) {
    cudaGetLastError();
    return fail(nullptr, MOE_ERR_CUDA, "no such CUDA device");
  }
  if (cudaSetDevice(cfg->device) != cudaSuccess) return fail(nullptr, MOE_ERR_CUDA, "cudaSetDevice failed");
  moe_handle* h = new moe_handle();
  h->cfg = *cfg;
  h->lay = moe::make_layout(cfg->wdtype, cfg->d, cfg->d_ff);
  h->slot_stride = align_up(h->lay.total, 256);
  h->n_gid = (int64_t)cfg->n_layers * cfg->n_experts;
  h->cap = slots_for(cfg, h->slot_stride);
  h->asize = cfg->adtype == MOE_DTYPE_FP32 ? 4 : 2;
  h->router_eb = cfg->wdtype == MOE_DTYPE_FP32 ? 4 : 2;
  const int64_t need = std::min<int64_t>(cfg->n_experts, (int64_t)cfg->top_k * cfg->max_batch);
  if (h->cap < need) {
    char buf[160];
    snprintf(buf, sizeof buf, "cap of %lld slots is below one layer-step's working set of %lld experts",
             (long long)h->cap, (long long)need);
    delete h;
    return fail(nullptr, MOE_ERR_CAPACITY, buf);
  }
  auto bail = [&](moe_status st, const std::string& msg) {
    const std::string keep = msg;  // msg may be h->err, which free_all destroys
    free_all(h);
    return fail(nullptr, st, keep);
  };
  if (cfg->device_pool) {
    if ((uintptr_t)cfg->device_pool % 256) return bail(MOE_ERR_INVALID, "device_pool must be 256-byte aligned");
    h->pool = (uint8_t*)cfg->device_pool;
  } else {
    if (cudaMalloc(&h->pool, h->cap * h->slot_stride) != cudaSuccess) {
      h->pool = nullptr;
      return bail(MOE_ERR_OOM, "device slot pool allocation failed");
    }
    h->own_pool = true;
  }
  {
    moe_status ast = alloc_arena(h);
    if (ast != MOE_OK) return bail(ast, h->err);
  }
  const int64_t rbytes = (int64_t)cfg->n_layers * cfg->n_experts * cfg->d * h->router_eb;
  if (cudaMalloc(&h->routers, rbytes) != cudaSuccess) return bail(MOE_ERR_OOM, "router allocation failed");
  if (cudaHostAlloc(&h->route, sizeof(moe::RouteOut), cudaHostAllocMapped) != cudaSuccess)
    return bail(MOE_ERR_OOM, "mapped routing buffer allocation failed");
  memset((void*)h->route, 0, sizeof(moe::RouteOut));
  h->route->seq = 0;
  if (cudaHostGetDevicePointer((void**)&h->route_dev, (void*)h->route, 0) != cudaSuccess)
    return bail(MOE_ERR_CUDA, "mapped routing buffer has no device address");
  // u per rank; the device lookahead kernel keeps the u of up to four groups of layers
  const int64_t u_sets = cfg->lookahead && cfg->schedule == MOE_SCHEDULE_DEVICE
                             ? std::max(4 * moe::kLaGroupMax, cfg->max_batch)
                             : cfg->max_batch;
  if (cudaMalloc(&h->u, sizeof(float) * u_sets * cfg->top_k * cfg->d_ff) != cudaSuccess)
    return bail(MOE_ERR_OOM, "u allocation failed");
  const int64_t act = (int64_t)cfg->n_layers * cfg->max_batch * cfg->d * h->asize;
  if (cudaMalloc(&h->hid_dev, act) != cudaSuccess || cudaMalloc(&h->out_dev, act) != cudaSuccess)
    return bail(MOE_ERR_OOM, "staging allocation failed");
  if (cudaStreamCreateWithFlags(&h->copy_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&h->host_stream, cudaStreamNonBlocking) != cudaSuccess)
    return bail(MOE_ERR_CUDA, "stream creation failed");
  h->copy_ev.resize((size_t)cfg->top_k * cfg->max_batch, nullptr);
  for (auto& e : h->copy_ev)
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return bail(MOE_ERR_CUDA, "event creation failed");
  for (auto& e : h->layer_ev)
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return bail(MOE_ERR_CUDA, "event creation failed");
  h->dev_mode = cfg->schedule == MOE_SCHEDULE_DEVICE;
  h->batched = h->dev_mode && cfg->max_batch > 1;
  h->batched_tc = h->batched && cfg->batched_path == MOE_BATCHED_AUTO &&
                  moe::batched_tc_supported(cfg->wdtype, cfg->d, cfg->d_ff);
  if (h->batched_tc) {
    h->fgrid = moe::fused_batched_tc_grid(cfg->d, cfg->d_ff, h->cap, h->n_gid);
    if (h->fgrid <= 0)
      return bail(MOE_ERR_INVALID, "cap not supported by the batched schedule (a cap that can evict must be at "
                                   "most 4096 slots)");
    moe_status ms = make_tc_maps(h);
    if (ms != MOE_OK) return bail(ms, h->err);
  } else if (h->batched) {
    h->fgrid = moe::fused_batched_grid(cfg->wdtype, cfg->d, cfg->d_ff, h->cap, h->n_gid);
    h->tg_max = moe::batched_tg(cfg->wdtype, cfg->d, cfg->d_ff);
    if (h->fgrid <= 0)
      return bail(MOE_ERR_INVALID, "shape or cap not supported by the batched schedule (a cap that can evict must be "
                                   "at most 4096 slots)");
  } else if (h->dev_mode) {
    h->fgrid = moe::fused_grid(cfg->wdtype, cfg->d, cfg->d_ff, cfg->top_k);
    if (h->fgrid <= 0) return bail(MOE_ERR_INVALID, "shape not supported by the device-driven schedule");
    if (cfg->lookahead) {
      // a miss must never take the slot of an expert the previous layer-step used (its down rows
      // may still be reading): LRU guarantees it from 2 k slots on
      const int64_t need_cap = 2 * (int64_t)cfg->top_k;
      if (h->cap < h->n_gid && h->cap < need_cap)
        return bail(MOE_ERR_INVALID, "lookahead in the device schedule needs at least " + std::to_string(need_cap) +
                                         " slots (or every expert resident)");
      // layers per worker barrier: a group of P layers needs a miss never to take the slot of an
      // expert of the 2 P - 1 layer-steps before it, which LRU guarantees from 2 P k slots on
      h->la_group = cfg->n_layers >= 2 && (h->cap >= h->n_gid || h->cap >= 2 * moe::kLaGroupMax * (int64_t)cfg->top_k)
                        ? moe::kLaGroupMax
                        : 1;
      h->fgrid_la = moe::fused_la_grid(cfg->wdtype, cfg->d, cfg->d_ff, cfg->top_k, h->la_group);
      if (h->fgrid_la <= 0 && h->la_group > 1) {
        h->la_group = 1;
        h->fgrid_la = moe::fused_la_grid(cfg->wdtype, cfg->d, cfg->d_ff, cfg->top_k, 1);
      }
      if (h->fgrid_la <= 0) return bail(MOE_ERR_INVALID, "shape not supported by the lookahead kernel");
      // Skewed workers (a group's down rows after the next group's gate/up rows) leave the down
      // rows of one more group reading while misses land: 3 P - 1 layer-steps before a miss's
      // own, kept by LRU from 3 P k slots on; with every expert resident nothing is evicted.
      h->la_skew = h->cap >= h->n_gid || h->cap >= 3 * (int64_t)h->la_group * cfg->top_k ? 1 : 0;
      h->lookahead_dev = true;
    }
  }
  if (h->dev_mode) {
    if (cudaHostGetDevicePointer((void**)&h->arena_dev, h->arena, 0) != cudaSuccess)
      return bail(MOE_ERR_CUDA, "host arena has no device address");
    const int k = cfg->top_k;
    const int64_t pairs = (int64_t)cfg->max_batch * k;
    // batch 1: slot, gid, miss per rank, for one layer ([k]) or, with lookahead, for every layer ([L][k])
    const int64_t plan_ranks = h->lookahead_dev ? (int64_t)k * cfg->n_layers : (int64_t)k;
    const int64_t plan_ints = h->batched ? 2 + 5 * (int64_t)cfg->n_experts + pairs : 3 * plan_ranks;
    bool ok = cudaMalloc(&h->d_slot_of, sizeof(int32_t) * h->n_gid) == cudaSuccess &&
              cudaMalloc(&h->d_slot_key, sizeof(unsigned long long) * h->cap) == cudaSuccess &&
              cudaMalloc(&h->d_cand, sizeof(unsigned long long) * (moe::kMaxRanks + 1)) == cudaSuccess &&
              cudaMalloc(&h->d_prior, sizeof(int32_t) * h->cap) == cudaSuccess &&
              cudaMalloc(&h->d_prior_slot_of, sizeof(int32_t) * h->n_gid) == cudaSuccess &&
              cudaMalloc(&h->d_rank, sizeof(int32_t) * h->n_gid) == cudaSuccess &&
              cudaMalloc(&h->d_rank_best, sizeof(int32_t) * 256) == cudaSuccess &&
              cudaMalloc(&h->d_hand, sizeof(int32_t)) == cudaSuccess &&
              cudaMalloc(&h->d_n_used, sizeof(int32_t)) == cudaSuccess &&
              cudaMalloc(&h->d_step, sizeof(int64_t)) == cudaSuccess &&
              cudaMalloc(&h->d_z, sizeof(float) * std::max<int64_t>(256 * (int64_t)cfg->max_batch,
                                                                    h->n_gid * cfg->max_batch)) == cudaSuccess &&
              cudaMalloc(&h->d_plan, sizeof(int32_t) * plan_ints) == cudaSuccess &&
              cudaMalloc(&h->d_plan_gate, sizeof(float) * std::max(pairs, plan_ranks)) == cudaSuccess &&
              (!h->batched || cudaMalloc(&h->d_sel_e, sizeof(int32_t) * pairs) == cudaSuccess) &&
              (!h->batched || cudaMalloc(&h->d_y, sizeof(float) * pairs * cfg->d) == cudaSuccess) &&
              cudaMalloc(&h->d_trace, sizeof(moe::TraceRec) * std::max<int64_t>(1, cfg->trace_capacity)) == cudaSuccess &&
              cudaMalloc(&h->d_trace_n, sizeof(unsigned long long)) == cudaSuccess &&
              cudaMalloc(&h->d_route_idx, sizeof(int32_t) * cfg->n_layers * pairs) == cudaSuccess &&
              cudaMalloc(&h->d_route_gate, sizeof(float) * cfg->n_layers * pairs) == cudaSuccess &&
              cudaMalloc(&h->d_stats, sizeof(unsigned long long) * moe::STAT_N) == cudaSuccess &&
              cudaMalloc(&h->d_bar, sizeof(unsigned) * 4) == cudaSuccess &&
              cudaMalloc(&h->d_err, sizeof(int)) == cudaSuccess &&
              cudaHostAlloc(&h->h_err, sizeof(int), cudaHostAllocDefault) == cudaSuccess &&
              cudaEventCreateWithFlags(&h->err_ev, cudaEventDisableTiming) == cudaSuccess;
    if (!ok) return bail(MOE_ERR_OOM, "device state allocation failed");
  }
  h->registered.assign(h->n_gid, 0);
  h->router_set.assign(cfg->n_layers, 0);
  h->table.init(h->n_gid, h->cap, cfg->policy, cfg->n_experts);
  if (cfg->trace_capacity > 0) h->trace.reserve((size_t)std::min<int64_t>(cfg->trace_capacity, 1 << 22));
  reset_state(h);
  *out = h;
  return MOE_OK;
}

moe_status moe_set_router(moe_handle* h, int32_t layer, const void* w_r) {
  if (!h) return MOE_ERR_INVALID;
  if (layer < 0 || layer >= h->cfg.n_layers || !w_r) return fail(h, MOE_ERR_INVALID, "bad layer or NULL weights");
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  const int64_t bytes = (int64_t)h->cfg.n_experts * h->cfg.d * h->router_eb;
  MOE_CK(h, cudaMemcpy(h->routers + layer * bytes, w_r, bytes, cudaMemcpyHostToDevice));
  h->router_set[layer] = 1;
  h->all_registered = false;
  return MOE_OK;
}

moe_status moe_register_host_experts(moe_handle* h, int32_t layer, int32_t expert, const void* w_gate,
                                     const void* w_up, const void* w_down, const void* scales) {
  if (!h) return MOE_ERR_INVALID;
  const moe_config& c = h->cfg;
  if (layer < 0 || layer >= c.n_layers || expert < 0 || expert >= c.n_experts)
    return fail(h, MOE_ERR_INVALID, "bad layer or expert id");
  if (!w_gate || !w_up || !w_down) return fail(h, MOE_ERR_INVALID, "NULL weight pointer");
  const bool q4 = c.wdtype == MOE_DTYPE_INT4_G128;
  if (q4 != (scales != nullptr)) return fail(h, MOE_ERR_INVALID, "scales must be given exactly for int4 weights");
  const int64_t gid = (int64_t)layer * c.n_experts + expert;
  uint8_t* dst = h->arena + gid * h->slot_stride;
  const moe::BlobLayout& L = h->lay;
  const int64_t rb = L.row_bytes_gu;
  const uint8_t* g = (const uint8_t*)w_gate;
  const uint8_t* u = (const uint8_t*)w_up;
  for (int64_t i = 0; i < c.d_ff; i++) {
    memcpy(dst + i * 2 * rb, g + i * rb, rb);
    memcpy(dst + i * 2 * rb + rb, u + i * rb, rb);
  }
  memcpy(dst + L.d_off, w_down, (size_t)(c.d * L.row_bytes_d));
  if (q4) {
    const int64_t G = c.d / 128;
    const uint16_t* s = (const uint16_t*)scales;
    uint16_t* gs = (uint16_t*)(dst + L.gu_scale_off);
    for (int64_t i = 0; i < c.d_ff; i++) {
      memcpy(gs + i * 2 * G, s + i * G, G * 2);
      memcpy(gs + i * 2 * G + G, s + c.d_ff * G + i * G, G * 2);
    }
    memcpy(dst + L.d_scale_off, s + 2 * c.d_ff * G, (size_t)(c.d * (c.d_ff / 128) * 2));
  }
  if (h->slot_stride > L.total) memset(dst + L.total, 0, h->slot_stride - L.total);
  h->registered[gid] = 1;
  return MOE_OK;
}

moe_status moe_decode_step(moe_handle* h, const void* hidden, void* out, int32_t batch, void* stream) {
  if (!h) return MOE_ERR_INVALID;
  if (!hidden || !out) return fail(h, MOE_ERR_INVALID, "NULL hidden or out");
  // the kernels move activation rows as 16-byte vectors: refuse a misaligned buffer here instead
  // of faulting the launch
  if ((((uintptr_t)hidden | (uintptr_t)out) & 15) != 0)
    return fail(h, MOE_ERR_INVALID, "hidden and out must be 16-byte aligned");
  if (batch < 1 || batch > h->cfg.max_batch) return fail(h, MOE_ERR_INVALID, "batch must be in [1, max_batch]");
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  moe_status st = check_registered(h);
  if (st != MOE_OK) return st;
  NvtxRange range(h->dev_mode ? "moe_decode_step (device schedule)" : "moe_decode_step (host schedule)");
  st = h->dev_mode ? decode_device(h, hidden, out, batch, (cudaStream_t)stream)
                   : decode_impl(h, hidden, out, (cudaStream_t)stream);
  if (st != MOE_OK) recover_after_failure(h, (cudaStream_t)stream);
  return st;
}

moe_status moe_decode_step_host(moe_handle* h, const void* hidden_host, void* out_host, int32_t batch) {
  if (!h) return MOE_ERR_INVALID;
  if (!hidden_host || !out_host) return fail(h, MOE_ERR_INVALID, "NULL hidden or out");
  if (batch < 1 || batch > h->cfg.max_batch) return fail(h, MOE_ERR_INVALID, "batch must be in [1, max_batch]");
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  NvtxRange range("moe_decode_step_host");
  const int64_t bytes = (int64_t)h->cfg.n_layers * batch * h->cfg.d * h->asize;
  MOE_CK(h, cudaMemcpyAsync(h->hid_dev, hidden_host, bytes, cudaMemcpyHostToDevice, h->host_stream));
  moe_status st = moe_decode_step(h, h->hid_dev, h->out_dev, batch, h->host_stream);
  if (st != MOE_OK) return st;
  MOE_CK(h, cudaMemcpyAsync(out_host, h->out_dev, bytes, cudaMemcpyDeviceToHost, h->host_stream));
  NvtxRange wait_range("wait for the step and its copies");
  MOE_CK(h, cudaStreamSynchronize(h->host_stream));
  return MOE_OK;
}

moe_status moe_get_residency_trace(moe_handle* h, int64_t start, moe_trace_rec* buf, int64_t cap, int64_t* n_copied,
                                   int64_t* n_total) {
  if (!h) return MOE_ERR_INVALID;
  if (start < 0 || cap < 0 || (cap > 0 && !buf)) return fail(h, MOE_ERR_INVALID, "bad trace range");
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  if (h->dev_mode) {
    moe_status st = check_device_error(h, true);
    if (st != MOE_OK) return st;
    unsigned long long produced = 0;
    MOE_CK(h, cudaMemcpy(&produced, h->d_trace_n, sizeof produced, cudaMemcpyDeviceToHost));
    const int64_t kept = std::min<int64_t>((int64_t)produced, h->cfg.trace_capacity);
    const int64_t n = std::max<int64_t>(0, std::min(cap, kept - start));
    if (n > 0) MOE_CK(h, cudaMemcpy(buf, h->d_trace + start, (size_t)n * sizeof(moe_trace_rec), cudaMemcpyDeviceToHost));
    if (n_copied) *n_copied = n;
    if (n_total) *n_total = kept;
    if ((int64_t)produced > kept) return fail(h, MOE_ERR_TRACE_OVERFLOW, "trace buffer full: records were dropped");
    return MOE_OK;
  }
  const int64_t tot = (int64_t)h->trace.size();
  const int64_t n = std::max<int64_t>(0, std::min(cap, tot - start));
  if (n > 0) memcpy(buf, h->trace.data() + start, (size_t)n * sizeof(moe_trace_rec));
  if (n_copied) *n_copied = n;
  if (n_total) *n_total = tot;
  if (h->trace_dropped > 0) return fail(h, MOE_ERR_TRACE_OVERFLOW, "trace buffer full: records were dropped");
  return MOE_OK;
}

moe_status moe_get_last_routing(moe_handle* h, int32_t* idx, float* gate, int64_t n) {
  if (!h) return MOE_ERR_INVALID;
  if (h->dev_mode) {
    const int64_t cnt = (int64_t)h->cfg.n_layers * h->cfg.max_batch * h->cfg.top_k;
    if (n < cnt) return fail(h, MOE_ERR_INVALID, "routing buffer too small");
    MOE_CK(h, cudaSetDevice(h->cfg.device));
    moe_status st = check_device_error(h, true);
    if (st != MOE_OK) return st;
    if (idx) MOE_CK(h, cudaMemcpy(idx, h->d_route_idx, cnt * sizeof(int32_t), cudaMemcpyDeviceToHost));
    if (gate) MOE_CK(h, cudaMemcpy(gate, h->d_route_gate, cnt * sizeof(float), cudaMemcpyDeviceToHost));
    return MOE_OK;
  }
  if (n < (int64_t)h->last_idx.size()) return fail(h, MOE_ERR_INVALID, "routing buffer too small");
  if (idx) memcpy(idx, h->last_idx.data(), h->last_idx.size() * sizeof(int32_t));
  if (gate) memcpy(gate, h->last_gate.data(), h->last_gate.size() * sizeof(float));
  return MOE_OK;
}

moe_status moe_get_last_logits(moe_handle* h, float* z, int64_t n) {
  if (!h || !z) return MOE_ERR_INVALID;
  const int64_t need = h->n_gid * h->cfg.max_batch;
  if (n < need) return fail(h, MOE_ERR_INVALID, "buffer below n_layers * max_batch * n_experts");
  if (!h->dev_mode) {
    if (h->cfg.policy != MOE_POLICY_GUIDED)
      return fail(h, MOE_ERR_INVALID, "the host schedule keeps router logits under the router-guided policy only");
    std::fill(z, z + need, 0.f);
    std::copy(h->last_z.begin(), h->last_z.end(), z);
    return MOE_OK;
  }
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  moe_status st = check_device_error(h, true);
  if (st != MOE_OK) return st;
  MOE_CK(h, cudaMemcpy(z, h->d_z, sizeof(float) * need, cudaMemcpyDeviceToHost));
  return MOE_OK;
}

moe_status moe_get_stats(moe_handle* h, moe_stats* out) {
  if (!h || !out) return MOE_ERR_INVALID;
  if (h->dev_mode) {
    MOE_CK(h, cudaSetDevice(h->cfg.device));
    moe_status st = check_device_error(h, true);
    if (st != MOE_OK) return st;
    unsigned long long v[moe::STAT_N];
    MOE_CK(h, cudaMemcpy(v, h->d_stats, sizeof v, cudaMemcpyDeviceToHost));
    out->steps = h->steps_launched;
    out->layer_steps = (int64_t)v[moe::STAT_LAYER_STEPS];
    out->hits = (int64_t)v[moe::STAT_HITS];
    out->misses = (int64_t)v[moe::STAT_MISSES];
    out->evictions = (int64_t)v[moe::STAT_EVICTIONS];
    out->miss_bytes = out->misses * h->lay.total;
    return MOE_OK;
  }
  *out = h->stats;
  return MOE_OK;
}

moe_status moe_reset_residency(moe_handle* h) {
  if (!h) return MOE_ERR_INVALID;
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  MOE_CK(h, cudaDeviceSynchronize());
  reset_state(h);
  return MOE_OK;
}

moe_status moe_preload(moe_handle* h, int64_t* n_loaded) {
  if (!h) return MOE_ERR_INVALID;
  NvtxRange range("moe_preload");
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  if (!h->all_registered) {
    for (int64_t g = 0; g < h->n_gid; g++)
      if (!h->registered[g]) return fail(h, MOE_ERR_NOT_REGISTERED, "preload needs every expert registered");
  }
  if (h->dev_mode) {
    moe_status st = check_device_error(h, true);
    if (st != MOE_OK) return st;
  } else {
    MOE_CK(h, cudaDeviceSynchronize());
  }
  if (!h->dev_mode) {
    // the host table decides the placements; a failed copy empties the pool again
    std::vector<std::pair<int32_t, int32_t>> placed;
    h->table.preload(placed);
    for (const auto& gs : placed) {
      cudaError_t e = cudaMemcpyAsync(h->pool + (int64_t)gs.second * h->slot_stride,
                                      h->arena + (int64_t)gs.first * h->slot_stride, h->lay.total,
                                      cudaMemcpyHostToDevice, h->copy_stream);
      if (e == cudaSuccess) continue;
      cudaStreamSynchronize(h->copy_stream);
      reset_state(h);
      return cuda_fail(h, e, "preload copy");
    }
    MOE_CK(h, cudaStreamSynchronize(h->copy_stream));
    if (n_loaded) *n_loaded = (int64_t)placed.size();
    return MOE_OK;
  }
  // device lookup table: free slots are [n_used, cap), filled in ascending gid
  std::vector<int32_t> slot_of(h->n_gid);
  int32_t n_used = 0;
  MOE_CK(h, cudaMemcpy(slot_of.data(), h->d_slot_of, sizeof(int32_t) * h->n_gid, cudaMemcpyDeviceToHost));
  MOE_CK(h, cudaMemcpy(&n_used, h->d_n_used, sizeof n_used, cudaMemcpyDeviceToHost));
  const bool guided = h->cfg.policy == MOE_POLICY_GUIDED;
  std::vector<int32_t> rank;
  if (guided) {
    rank.resize(h->n_gid);
    MOE_CK(h, cudaMemcpy(rank.data(), h->d_rank, sizeof(int32_t) * h->n_gid, cudaMemcpyDeviceToHost));
  }
  int64_t loaded = 0;
  std::vector<unsigned long long> keys;
  std::vector<int32_t> kslots;
  for (int64_t g = 0; g < h->n_gid && n_used < h->cap; g++) {
    if (slot_of[g] >= 0) continue;
    const int32_t slot = n_used++;
    MOE_CK(h, cudaMemcpyAsync(h->pool + (int64_t)slot * h->slot_stride, h->arena + g * h->slot_stride, h->lay.total,
                              cudaMemcpyHostToDevice, h->copy_stream));
    slot_of[g] = slot;
    // last use 0: older than every decode step
    keys.push_back(guided ? moe::guided_key(h->cfg.n_experts, rank[g], 0u, (int32_t)g) : (unsigned long long)(uint32_t)g);
    kslots.push_back(slot);
    loaded++;
  }
  MOE_CK(h, cudaStreamSynchronize(h->copy_stream));
  if (loaded > 0) {
    MOE_CK(h, cudaMemcpy(h->d_slot_of, slot_of.data(), sizeof(int32_t) * h->n_gid, cudaMemcpyHostToDevice));
    MOE_CK(h, cudaMemcpy(h->d_n_used, &n_used, sizeof n_used, cudaMemcpyHostToDevice));
    // preloaded slots are contiguous [n_used - loaded, n_used)
    MOE_CK(h, cudaMemcpy(h->d_slot_key + kslots.front(), keys.data(), sizeof(unsigned long long) * keys.size(),
                         cudaMemcpyHostToDevice));
    MOE_CK(h, cudaMemset(h->d_cand, 0, sizeof(unsigned long long) * (moe::kMaxRanks + 1)));  // keys changed
  }
  if (n_loaded) *n_loaded = loaded;
  return MOE_OK;
}

moe_status moe_profile_enable(moe_handle* h, int32_t on) {
  if (!h) return MOE_ERR_INVALID;
  h->prof = on != 0;
  return MOE_OK;
}

moe_status moe_profile_read(moe_handle* h, moe_kernel_time* out, int32_t cap, int32_t* n_out) {
  if (!h || (cap > 0 && !out)) return MOE_ERR_INVALID;
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  harvest(h, true);
  int32_t n = 0;
  for (int c = 0; c < PC_N && n < cap; c++, n++) {  // fused_phase_*: per layer-step, from the kernel's global timer
    memset(&out[n], 0, sizeof(moe_kernel_time));
    snprintf(out[n].name, sizeof out[n].name, "%s", kPcName[c]);
    out[n].launches = h->pc_launches[c];
    out[n].total_ms = h->pc_ms[c];
    out[n].bytes = h->pc_bytes[c];
    h->pc_launches[c] = 0;
    h->pc_ms[c] = 0;
    h->pc_bytes[c] = 0;
  }
  if (n_out) *n_out = n;
  return MOE_OK;
}

const char* moe_last_error(const moe_handle* h) { return h ? h->err.c_str() : g_create_error.c_str(); }

moe_status moe_inject_fault(moe_handle* h, int32_t kind) {
  if (!h) return MOE_ERR_INVALID;
  if (kind == MOE_FAULT_BARRIER_TIMEOUT && !h->dev_mode)
    return fail(h, MOE_ERR_INVALID, "barrier faults need the device schedule");
  if (kind == MOE_FAULT_COPY_ERROR && h->dev_mode)
    return fail(h, MOE_ERR_INVALID, "copy faults need the host copy-engine schedule");
  if (kind != MOE_FAULT_NONE && kind != MOE_FAULT_BARRIER_TIMEOUT && kind != MOE_FAULT_COPY_ERROR)
    return fail(h, MOE_ERR_INVALID, "unknown fault kind");
  h->fault = kind;
  return MOE_OK;
}

void moe_destroy(moe_handle* h) {
  if (!h) return;
  cudaSetDevice(h->cfg.device);
  free_all(h);
}

}  // extern "C"

namespace moe {

bool moe_shape(const moe_handle* h, MoeShape* out) {
  if (!h || !out) return false;
  const moe_config& c = h->cfg;
  out->d = c.d;
  out->n_layers = c.n_layers;
  out->top_k = c.top_k;
  out->n_experts = c.n_experts;
  out->wdtype = c.wdtype;
  out->adtype = c.adtype;
  out->device = c.device;
  out->device_batch1 = h->dev_mode && !h->batched && c.max_batch == 1;
  return true;
}

moe_status moe_run_layer(moe_handle* h, const void* hidden, void* out, int32_t layer, cudaStream_t s) {
  if (!h) return MOE_ERR_INVALID;
  if (!h->dev_mode || h->batched) return fail(h, MOE_ERR_INVALID, "a chained decoder needs the batch-1 device schedule");
  if (layer < 0 || layer >= h->cfg.n_layers) return fail(h, MOE_ERR_INVALID, "layer out of range");
  MOE_CK(h, cudaSetDevice(h->cfg.device));
  moe_status st = MOE_OK;
  if (layer == 0) {
    st = check_registered(h);
    if (st != MOE_OK) return st;
    st = check_device_error(h, false);
    if (st != MOE_OK) return st;
    st = rewarm_if_idle(h, s);  // once per decoder token, before its first MoE layer
    if (st != MOE_OK) return st;
  }
  st = decode_device_layers(h, hidden, out, layer, layer + 1, s);
  if (st != MOE_OK) recover_after_failure(h, s);
  return st;
}

const char* moe_error_text(const moe_handle* h) { return h ? h->err.c_str() : ""; }

}  // namespace moe
