// Residency planner (C ABI declared in moe.h): the library's host slot table driven by expert
// selections the caller supplies. No GPU, no weights, no copies: it answers which experts a given
// routing sequence would hit, miss, evict or prefetch under a cap and a policy, with the decisions
// the host-driven decode schedule makes.
#include <algorithm>
#include <cstdint>
#include <new>
#include <string>
#include <vector>

#include "moe.h"
#include "slot_table.h"

struct moe_planner {
  int32_t n_layers = 0, n_experts = 0;
  moe::SlotTable table;
  int64_t last_step = -1;
  int32_t last_layer = -1;
  bool broken = false;
  std::vector<int32_t> needed, cand;
  std::vector<moe::SlotDecision> dec;
  std::string err;
};

namespace {

thread_local std::string g_planner_create_error;

moe_status planner_fail(moe_planner* p, moe_status st, const char* msg) {
  p->err = msg;
  return st;
}

// Distinct ids of one layer, ascending, as global ids; false if one is out of range.
bool gather_ids(const int32_t* ids, int32_t n, int32_t layer, int32_t E, std::vector<int32_t>& out) {
  out.clear();
  for (int32_t i = 0; i < n; i++) {
    if (ids[i] < 0 || ids[i] >= E) return false;
    out.push_back(layer * E + ids[i]);
  }
  std::sort(out.begin(), out.end());
  out.erase(std::unique(out.begin(), out.end()), out.end());
  return true;
}

}  // namespace

extern "C" {

moe_status moe_planner_create(int32_t n_layers, int32_t n_experts, int64_t cap_slots, int32_t policy,
                              moe_planner** out) {
  if (!out) return MOE_ERR_INVALID;
  *out = nullptr;
  const char* bad = nullptr;
  if (n_layers < 1 || n_experts < 1)
    bad = "n_layers and n_experts must be at least 1";
  else if ((int64_t)n_layers * n_experts > INT32_MAX)
    bad = "n_layers * n_experts must fit in int32";
  else if (cap_slots < 1 || cap_slots > INT32_MAX)
    bad = "cap_slots must be in [1, 2^31)";
  else if (policy != MOE_POLICY_LRU && policy != MOE_POLICY_ROTARY && policy != MOE_POLICY_GUIDED)
    bad = "unknown policy";
  if (bad) {
    g_planner_create_error = bad;
    return MOE_ERR_INVALID;
  }
  moe_planner* p = new (std::nothrow) moe_planner();
  if (!p) {
    g_planner_create_error = "host allocation failed";
    return MOE_ERR_OOM;
  }
  const int64_t n_gid = (int64_t)n_layers * n_experts;
  try {
    p->table.init(n_gid, std::min(cap_slots, n_gid), policy, n_experts);
  } catch (const std::bad_alloc&) {
    delete p;
    g_planner_create_error = "host allocation failed";
    return MOE_ERR_OOM;
  }
  p->n_layers = n_layers;
  p->n_experts = n_experts;
  *out = p;
  return MOE_OK;
}

moe_status moe_planner_preload(moe_planner* p, int64_t* n_loaded) {
  if (!p) return MOE_ERR_INVALID;
  if (p->broken) return planner_fail(p, MOE_ERR_INVALID, "the planner failed a step earlier");
  std::vector<std::pair<int32_t, int32_t>> placed;
  try {
    p->table.preload(placed);
  } catch (const std::bad_alloc&) {
    p->broken = true;
    return planner_fail(p, MOE_ERR_OOM, "host allocation failed");
  }
  if (n_loaded) *n_loaded = (int64_t)placed.size();
  return MOE_OK;
}

moe_status moe_planner_step(moe_planner* p, int64_t step, int32_t layer, const int32_t* experts, int32_t n,
                            const int32_t* prefetch, int32_t n_prefetch, const int32_t* ranks, moe_trace_rec* recs,
                            int32_t recs_cap, int32_t* n_recs) {
  if (!p) return MOE_ERR_INVALID;
  if (n_recs) *n_recs = 0;
  if (p->broken) return planner_fail(p, MOE_ERR_INVALID, "the planner failed a step earlier");
  if (step < 0 || step > INT32_MAX || layer < 0 || layer >= p->n_layers)
    return planner_fail(p, MOE_ERR_INVALID, "step must be in [0, 2^31) and layer in [0, n_layers)");
  if (step < p->last_step || (step == p->last_step && layer <= p->last_layer))
    return planner_fail(p, MOE_ERR_INVALID, "layer-steps must come in increasing (step, layer) order");
  if (n < 0 || n_prefetch < 0 || (n > 0 && !experts) || (n_prefetch > 0 && !prefetch) || !recs || !n_recs)
    return planner_fail(p, MOE_ERR_INVALID, "bad counts or NULL buffers");
  if (n_prefetch > 0 && p->table.policy() != MOE_POLICY_LRU)
    return planner_fail(p, MOE_ERR_INVALID, "prefetch admission is defined for the LRU policy only");
  if ((int64_t)recs_cap < (int64_t)n + n_prefetch)
    return planner_fail(p, MOE_ERR_INVALID, "recs_cap below n + n_prefetch");
  const int32_t E = p->n_experts;
  const bool guided = p->table.policy() == MOE_POLICY_GUIDED;
  if (guided != (ranks != nullptr))
    return planner_fail(p, MOE_ERR_INVALID, "ranks are required by the guided policy and taken by no other");
  if (guided) {
    for (int32_t e = 0; e < E; e++)
      if (ranks[e] < 0 || ranks[e] > E) return planner_fail(p, MOE_ERR_INVALID, "a rank is outside [0, n_experts]");
  }
  bool ok = false;
  try {
    if (!gather_ids(experts, n, layer, E, p->needed) || !gather_ids(prefetch, n_prefetch, layer, E, p->cand))
      return planner_fail(p, MOE_ERR_INVALID, "an expert id is outside [0, n_experts)");
    const int64_t clock = step * p->n_layers + layer + 1;  // 0: preloaded, older than every step
    p->dec.clear();
    if (guided) p->table.set_ranks(layer, ranks);
    ok = p->table.step(p->needed.data(), (int32_t)p->needed.size(), clock, p->dec);
    if (ok && !p->cand.empty())
      p->table.admit(p->needed.data(), (int32_t)p->needed.size(), p->cand.data(), (int32_t)p->cand.size(), clock,
                     p->dec);
  } catch (const std::bad_alloc&) {
    p->broken = true;
    return planner_fail(p, MOE_ERR_OOM, "host allocation failed");
  }
  for (size_t i = 0; i < p->dec.size(); i++) {
    const moe::SlotDecision& d = p->dec[i];
    recs[i] = moe_trace_rec{(int32_t)step, layer, d.gid - layer * E, d.kind, d.slot, d.evicted};
  }
  *n_recs = (int32_t)p->dec.size();
  p->last_step = step;
  p->last_layer = layer;
  if (!ok) {
    p->broken = true;
    return planner_fail(p, MOE_ERR_CAPACITY, "no slot available (cap below the layer-step's working set)");
  }
  return MOE_OK;
}

const char* moe_planner_last_error(const moe_planner* p) {
  return p ? p->err.c_str() : g_planner_create_error.c_str();
}

void moe_planner_destroy(moe_planner* p) { delete p; }

}  // extern "C"
