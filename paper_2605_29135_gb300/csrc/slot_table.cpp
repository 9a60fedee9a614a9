// Host residency table (rules in slot_table.h).
#include "slot_table.h"

#include <algorithm>

#include "moe.h"

namespace moe {

void SlotTable::init(int64_t n_gid, int64_t cap, int32_t policy, int32_t n_experts) {
  n_gid_ = n_gid;
  cap_ = cap;
  policy_ = policy;
  n_experts_ = n_experts;
  reset();
}

void SlotTable::reset() {
  slot_of_.assign(n_gid_, -1);
  gid_of_.assign(cap_, -1);
  last_use_.assign(n_gid_, -1);
  mark_.assign(n_gid_, 0);
  lru_.clear();
  free_.clear();
  for (int64_t s = 0; s < cap_; s++) free_.insert((int32_t)s);
  prior_.assign(cap_, -1);
  prior_slot_of_.assign(n_gid_, -1);
  hand_ = 0;
  rank_.assign(n_gid_, n_experts_);
}

void SlotTable::set_ranks(int32_t layer, const int32_t* ranks) {
  std::copy(ranks, ranks + n_experts_, rank_.begin() + (int64_t)layer * n_experts_);
}

int32_t SlotTable::take_free() {
  const int32_t s = *free_.begin();
  free_.erase(free_.begin());
  return s;
}

int32_t SlotTable::lru_victim() {
  for (auto it = lru_.begin(); it != lru_.end(); ++it) {
    if (!mark_[it->second]) {
      const int32_t v = it->second;
      lru_.erase(it);
      return v;
    }
  }
  return -1;
}

int32_t SlotTable::guided_victim() {
  int32_t victim = -1;
  for (int64_t s = 0; s < cap_; s++) {
    const int32_t v = gid_of_[s];
    if (v < 0 || mark_[v]) continue;
    if (victim < 0 || rank_[v] > rank_[victim] ||
        (rank_[v] == rank_[victim] &&
         (last_use_[v] > last_use_[victim] || (last_use_[v] == last_use_[victim] && v < victim))))
      victim = v;
  }
  return victim;
}

bool SlotTable::step(const int32_t* needed, int32_t n, int64_t clock, std::vector<SlotDecision>& out) {
  for (int32_t i = 0; i < n; i++) mark_[needed[i]] = 1;
  bool ok = true;
  const size_t first = out.size();
  for (int32_t i = 0; i < n; i++) {
    const int32_t g = needed[i];
    if (slot_of_[g] >= 0) {
      out.push_back(SlotDecision{g, SLOT_HIT, slot_of_[g], -1});
      continue;
    }
    int32_t slot = -1, victim = -1;
    if (policy_ == MOE_POLICY_ROTARY) {
      auto open = [&](int32_t s) { return gid_of_[s] < 0 || !mark_[gid_of_[s]]; };
      const int32_t ps = prior_slot_of_[g];
      if (ps >= 0 && open(ps)) slot = ps;
      if (slot < 0) {
        for (int64_t j = 0; j < cap_; j++) {
          const int32_t sj = (int32_t)((hand_ + j) % cap_);
          if (open(sj)) {
            slot = sj;
            break;
          }
        }
        if (slot < 0) {
          ok = false;
          break;
        }
        hand_ = (slot + 1) % cap_;
      }
      victim = gid_of_[slot];
      if (victim >= 0)
        slot_of_[victim] = -1;
      else
        free_.erase(slot);
      if (ps >= 0) prior_[ps] = -1;  // g is no longer anyone's prior occupant
      const int32_t u = prior_[slot];
      if (u >= 0) prior_slot_of_[u] = -1;
      prior_[slot] = victim;
      if (victim >= 0) prior_slot_of_[victim] = slot;
      prior_slot_of_[g] = -1;
    } else if (!free_.empty()) {
      slot = take_free();
    } else {
      victim = policy_ == MOE_POLICY_GUIDED ? guided_victim() : lru_victim();
      if (victim < 0) {
        ok = false;
        break;
      }
      slot = slot_of_[victim];
      slot_of_[victim] = -1;
    }
    gid_of_[slot] = g;
    slot_of_[g] = slot;
    out.push_back(SlotDecision{g, SLOT_MISS, slot, victim});
  }
  for (int32_t i = 0; i < n; i++) mark_[needed[i]] = 0;
  if (!ok || policy_ == MOE_POLICY_ROTARY) return ok;
  for (int32_t i = 0; i < n; i++) {
    const int32_t g = needed[i];
    if (policy_ == MOE_POLICY_LRU && out[first + i].kind == SLOT_HIT) lru_.erase({last_use_[g], g});
    last_use_[g] = clock;
    if (policy_ == MOE_POLICY_LRU) lru_.insert({clock, g});
  }
  return true;
}

void SlotTable::admit(const int32_t* needed, int32_t n, const int32_t* cand, int32_t m, int64_t clock,
                      std::vector<SlotDecision>& out) {
  if (policy_ != MOE_POLICY_LRU) return;
  for (int32_t i = 0; i < n; i++) mark_[needed[i]] = 1;
  for (int32_t i = 0; i < m; i++) mark_[cand[i]] = 1;
  for (int32_t i = 0; i < m; i++) {
    const int32_t g = cand[i];
    if (slot_of_[g] >= 0) continue;
    int32_t slot = -1, victim = -1;
    if (!free_.empty()) {
      slot = take_free();
    } else {
      victim = lru_victim();
      if (victim < 0) break;
      slot = slot_of_[victim];
      slot_of_[victim] = -1;
    }
    gid_of_[slot] = g;
    slot_of_[g] = slot;
    last_use_[g] = clock;
    lru_.insert({clock, g});
    out.push_back(SlotDecision{g, SLOT_PREFETCH, slot, victim});
  }
  for (int32_t i = 0; i < n; i++) mark_[needed[i]] = 0;
  for (int32_t i = 0; i < m; i++) mark_[cand[i]] = 0;
}

void SlotTable::preload(std::vector<std::pair<int32_t, int32_t>>& placed) {
  int64_t g = 0;
  while (!free_.empty()) {
    while (g < n_gid_ && slot_of_[g] >= 0) g++;
    if (g >= n_gid_) break;
    const int32_t slot = take_free();
    gid_of_[slot] = (int32_t)g;
    slot_of_[g] = slot;
    last_use_[g] = 0;
    lru_.insert({0, (int32_t)g});
    placed.emplace_back((int32_t)g, slot);
    g++;
  }
}

}  // namespace moe
