// Host residency table: a fixed group of `cap` slots, the lookup table global expert id -> slot
// and its replacement policy (paper Sec. 3, Fig. 1: slot group, lookup table, selective load and
// evict driven by the routing result). The host-driven decode schedule and the residency planner
// both run this code; the device schedule applies the LRU and rotary rules inside its kernel.
//
// Rules of one layer-step (needed: the distinct global ids the step uses, ascending):
//   LRU (MOE_POLICY_LRU): a resident id is a hit. A missing id takes the lowest free slot, else
//     the slot of the resident with the smallest (last use, id) that the step does not need.
//     Every needed id then gets the step's clock as its last use.
//   Rotary (MOE_POLICY_ROTARY): the slots form a ring with a hand and each slot remembers the id
//     last evicted from it. A missing id returns to the slot it was last evicted from when that
//     slot holds nothing the step needs (reverse rotation), else takes the first such slot at or
//     after the hand, which then moves past it (forward rotation). Hits change nothing.
//   Router-guided (MOE_POLICY_GUIDED): each id carries its rank in its layer's most recent routing
//     (set_ranks, before the layer's step; n_experts until the layer is first routed). A missing
//     id takes the lowest free slot, else the slot of the resident the step does not need with the
//     largest rank, ties to the larger (more recent) last use, then to the lower id. Every needed
//     id then gets the step's clock as its last use.
// Prefetch admission (LRU only; one reading of the paper's residency decisions that use
// information produced during execution, Sec. 3): after a step, candidate ids (ascending) that are
// absent take the lowest free slot, else the slot of the resident with the smallest (last use, id)
// outside the step's needed ids and the candidates; when none is left the rest are dropped. An
// admitted id gets the step's clock; a candidate already resident is left as it is.
#pragma once
#include <cstdint>
#include <set>
#include <utility>
#include <vector>

namespace moe {

enum : int32_t { SLOT_HIT = 0, SLOT_MISS = 1, SLOT_PREFETCH = 2 };

struct SlotDecision {
  int32_t gid;
  int32_t kind;     // SLOT_HIT, SLOT_MISS or SLOT_PREFETCH
  int32_t slot;     // slot that holds gid afterwards
  int32_t evicted;  // id evicted from that slot, -1 when none
};

class SlotTable {
 public:
  // policy: MOE_POLICY_LRU, MOE_POLICY_ROTARY or MOE_POLICY_GUIDED; ids are layer * n_experts +
  // expert. Starts empty.
  void init(int64_t n_gid, int64_t cap, int32_t policy, int32_t n_experts);
  // Every slot free, hand at slot 0, no remembered occupants, no layer routed.
  void reset();

  // Router-guided policy: ranks [n_experts] of the layer's experts in its latest routing.
  void set_ranks(int32_t layer, const int32_t* ranks);

  // One layer-step: appends one decision per needed id (ascending, distinct, in [0, n_gid)).
  // Returns false when a missing id finds no slot (cap below the step's working set); the
  // decisions made so far stay applied and appended, and no last use is updated.
  bool step(const int32_t* needed, int32_t n, int64_t clock, std::vector<SlotDecision>& out);

  // Prefetch admission right after step(needed, clock): appends one SLOT_PREFETCH decision per
  // admitted candidate. cand: ascending, distinct, in [0, n_gid). LRU only (no-op otherwise).
  void admit(const int32_t* needed, int32_t n, const int32_t* cand, int32_t m, int64_t clock,
             std::vector<SlotDecision>& out);

  // Warm start: free slots (lowest first) take absent ids in ascending order until none is free.
  // Placed ids count as used before every step (last use 0; steps use clocks >= 1). Appends the
  // (gid, slot) placements.
  void preload(std::vector<std::pair<int32_t, int32_t>>& placed);

  int32_t slot_of(int32_t gid) const { return slot_of_[gid]; }
  int32_t gid_of(int64_t slot) const { return gid_of_[slot]; }
  int64_t n_gid() const { return n_gid_; }
  int64_t cap() const { return cap_; }
  int32_t policy() const { return policy_; }
  int64_t n_free() const { return (int64_t)free_.size(); }

 private:
  int32_t take_free();
  int32_t lru_victim();     // resident with the smallest (last use, id) not marked; -1 when none
  int32_t guided_victim();  // resident with the largest (rank, last use, -id) not marked; -1 when none

  int64_t n_gid_ = 0, cap_ = 0;
  int32_t policy_ = 0;
  int32_t n_experts_ = 1;
  std::vector<int32_t> rank_;  // router-guided policy: [n_gid]
  std::vector<int32_t> slot_of_, gid_of_;
  std::vector<int64_t> last_use_;
  std::vector<uint8_t> mark_;                  // needed (or admitted) in the current call
  std::set<std::pair<int64_t, int32_t>> lru_;  // residents as (last use, id)
  std::set<int32_t> free_;
  // rotary slot group
  std::vector<int32_t> prior_;          // [cap]: id last evicted from the slot, -1 none
  std::vector<int32_t> prior_slot_of_;  // [n_gid]: the slot whose prior occupant is the id, -1 none
  int64_t hand_ = 0;
};

}  // namespace moe
