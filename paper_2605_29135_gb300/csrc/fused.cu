// Device-driven decode step (sm_103a): one cooperative persistent kernel per decode step.
//
// Per layer, phases R, C and D are separated by grid barriers; phase S runs in CTA 0 alongside
// the start of phase C. Every CTA repeats the layer's top-k and classifies the selected experts
// as hits or misses from the lookup table as it was before the step (S holds its table writes
// back until phase D), so the hit rows of phase C start right after R; only the miss CTAs wait
// (bounded) for CTA 0's published plan, which holds the misses' slots.
//   R  router logits z = W_r h, one warp per expert row;
//   S  CTA 0: top-k (ties -> lower id) and gates, then one step of the lookup table: hits keep
//      their slot, misses (ascending global id) take the lowest free slot, else the unpinned
//      resident with the smallest key: (last use, global id) under LRU; under router-guided
//      replacement the largest rank in its layer's latest routing first (this layer's ranks are
//      refreshed from z before the lookup), then the most recent use; the rotary ring otherwise.
//      Records go to the trace buffer and the per-rank plan (slot, miss flag, gate) to global
//      memory;
//   C  gate-up rows of every rank, u_r[i] = silu(W_g[i] . h) * (W_u[i] . h). A few "miss CTAs"
//      stream every missed expert from the page-locked host tier over NVLink-C2C: its gate/up
//      rows are stored into the freed slot and used for u in the same pass, and its W_d region
//      is copied into the slot; the other CTAs compute the hit experts' rows from HBM at the
//      same time. Capping the warps that read the host tier keeps the link's outstanding
//      requests near what saturates it (tens of warps, not thousands);
//   D  down rows + combine from the slots, out[o] = sum_r g_r (W_d^(r)[o] . u_r) in rank order.
//
// All CTAs are co-resident (cooperative launch). Every barrier wait, and the miss CTAs' wait for
// the plan, is bounded by a timeout on the global timer; on expiry the kernel sets an error flag
// and every CTA returns.
#include <cuda_bf16.h>
#include <math.h>

#include "dev.cuh"
#include "fused.cuh"
#include "grid.cuh"
#include "topk.cuh"

namespace moe {
namespace {

using namespace dev;

constexpr int kFWarps = 8;
constexpr int kFThreads = kFWarps * 32;

__device__ __forceinline__ unsigned long long shfl_min_u64(unsigned long long v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const unsigned long long o = __shfl_xor_sync(kFull, v, off);
    v = o < v ? o : v;
  }
  return v;
}

// The k smallest slot keys of a full pool, ascending, into a.cand (CTA 0, all threads; keys are
// distinct, so round j takes the smallest key above round j - 1's).
__device__ void find_victim_candidates(const FusedArgs& a) {
  __shared__ unsigned long long s_min[kFWarps];
  __shared__ unsigned long long s_last;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  unsigned long long last = 0ull;
  for (int j = 0; j < a.k; j++) {
    unsigned long long best = ~0ull;
    for (int64_t sl = threadIdx.x; sl < a.cap; sl += blockDim.x) {
      const unsigned long long key = __ldcg(a.slot_key + sl);
      if ((j == 0 || key > last) && key < best) best = key;
    }
    best = shfl_min_u64(best);
    if (lane == 0) s_min[warp] = best;
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned long long m = s_min[0];
      for (int w = 1; w < kFWarps; w++) m = s_min[w] < m ? s_min[w] : m;
      a.cand[j] = m;
      s_last = m;
    }
    __syncthreads();
    last = s_last;
  }
  if (threadIdx.x == 0) a.cand[kMaxRanks] = (unsigned long long)a.k;
}

// Lookup-table writes of a layer-step, held back until phase D: during phase C every CTA classifies
// the layer's selected experts as hits or misses from the table as it was before the step, while
// CTA 0 is still deciding the step (thread 0 of CTA 0 records, the same thread applies).
struct PendingTable {
  int n;
  int gid[2 * kMaxRanks];
  int val[2 * kMaxRanks];
  __device__ void set(int g, int v) {
    gid[n] = g;
    val[n] = v;
    n++;
  }
  __device__ void apply(const FusedArgs& a) {
    for (int i = 0; i < n; i++) a.slot_of[gid[i]] = val[i];
    n = 0;
  }
};

// Rotary slot-group step for the misses of one layer-step (thread 0 of CTA 0; at most k misses,
// in ascending id). A miss returns to the slot it was last evicted from when that slot holds no
// expert of the step (reverse rotation), else takes the first such slot at or after the hand, which
// moves past it (forward rotation). Uses what phase S read up front: the layer's previous-slot
// entries with those slots' occupants, and the min(cap, 2k + 1) slots from the hand (a step skips
// at most k pinned slots and takes at most k), updated here as the step places experts.
__device__ void rotary_place(const FusedArgs& a, int l, int clock, int k, int E, const int* need, const int* miss,
                             int* slot_out, int* evict_out, const int* ps_e, const int* ps_gid, int* win_gid,
                             int* win_prior, int hand0, int nused0, PendingTable& pend) {
  const int nw = 2 * k + 1 < a.cap ? 2 * k + 1 : (int)a.cap;
  int placed_slot[kMaxRanks], placed_gid[kMaxRanks];
  int np = 0;
  auto in_need = [&](int g) {
    bool f = false;
    for (int t = 0; t < k; t++) f |= need[t] == g;
    return f;
  };
  auto win_index = [&](int sl) {  // position of slot sl in the window, -1 outside
    const int j = (int)(((int64_t)sl - hand0 + a.cap) % a.cap);
    return j < nw ? j : -1;
  };
  int hand = hand0, nused = nused0;
  unsigned long long misses = 0, evictions = 0;
  for (int t = 0; t < k; t++) {
    if (!miss[t]) continue;
    misses++;
    const int g = need[t];
    const int e = g - l * E;
    // current occupant of a slot: this step's placements first, then what was read up front
    auto occupant = [&](int sl, int fallback) {
      int o = fallback;
      for (int q = 0; q < np; q++)
        if (placed_slot[q] == sl) o = placed_gid[q];
      return o;
    };
    int slot = -1, occ = -1;
    // g's return slot, while that slot's previous occupant is still g (an earlier miss of this
    // step may have taken the slot; slots outside the window change only by a return of g itself)
    int ps = ps_e[e];
    if (ps >= 0) {
      const int wj = win_index(ps);
      if (wj >= 0 && win_prior[wj] != g) ps = -1;
    }
    if (ps >= 0) {
      const int wj = win_index(ps);
      const int o = occupant(ps, wj >= 0 ? win_gid[wj] : ps_gid[e]);
      if (o < 0 || !in_need(o)) {
        slot = ps;
        occ = o;
      }
    }
    if (slot < 0) {
      for (int j = 0; j < nw; j++) {
        const int sl = (int)((hand + (int64_t)j) % a.cap);
        const int wj = win_index(sl);
        if (wj < 0) break;  // cannot happen (see above); reported as no available slot
        const int o = occupant(sl, win_gid[wj]);
        if (o < 0 || !in_need(o)) {
          slot = sl;
          occ = o;
          break;
        }
      }
      if (slot < 0) {
        atomicOr(a.err, FERR_NO_VICTIM);
        slot_out[t] = -1;
        continue;
      }
      hand = (int)((slot + 1) % a.cap);
    }
    // evict the occupant; bookkeeping of previous occupants
    if (occ >= 0) {
      pend.set(occ, -1);
      evictions++;
    } else {
      nused++;
    }
    if (ps >= 0) {
      a.prior[ps] = -1;
      const int wj = win_index(ps);
      if (wj >= 0) win_prior[wj] = -1;
    }
    const int wj = win_index(slot);
    const int u = slot == ps ? -1 : (wj >= 0 ? win_prior[wj] : -1);
    if (u >= 0) a.prior_slot_of[u] = -1;
    a.prior[slot] = occ;
    if (wj >= 0) win_prior[wj] = occ;
    if (occ >= 0) a.prior_slot_of[occ] = slot;
    a.prior_slot_of[g] = -1;
    pend.set(g, slot);
    placed_slot[np] = slot;
    placed_gid[np] = g;
    np++;
    slot_out[t] = slot;
    evict_out[t] = occ;
  }
  for (int t = 0; t < k; t++)
    if (slot_out[t] >= 0) a.slot_key[slot_out[t]] = ((unsigned long long)(uint32_t)clock << 32) | (uint32_t)need[t];
  if (hand != hand0) *a.hand = hand;
  if (nused != nused0) *a.n_used = nused;
  atomicAdd(a.stats + STAT_HITS, (unsigned long long)k - misses);
  atomicAdd(a.stats + STAT_MISSES, misses);
  atomicAdd(a.stats + STAT_EVICTIONS, evictions);
  atomicAdd(a.stats + STAT_LAYER_STEPS, 1ull);
}

// Phase S, run by CTA 0 (all its threads). Every global read the phase needs is issued at its
// start, side by side: the logits (warp 0), the layer's row of the lookup table, the pool's fill
// count, the trace position and the victim candidates (warps 1-7).
__device__ void select_and_lookup(const FusedArgs& a, int l, int clock, int64_t step, PendingTable& pend,
                                  int64_t po = 0) {
  __shared__ int s_idx[kMaxRanks];
  __shared__ float s_gate[kMaxRanks];
  __shared__ int s_need[kMaxRanks];   // needed global ids, ascending
  __shared__ int s_slot[kMaxRanks];   // slot per needed id (after the step)
  __shared__ int s_miss[kMaxRanks];
  __shared__ int s_evict[kMaxRanks];  // evicted global id per needed id, -1 if none
  __shared__ int s_vslot[kMaxRanks];  // victims in ascending (last use, id): slot and global id
  __shared__ int s_vgid[kMaxRanks];
  __shared__ int s_nev, s_nev_found, s_nused, s_ncand;
  __shared__ unsigned long long s_trace_base;
  __shared__ int s_slot_e[256];       // the layer's row of the lookup table
  __shared__ int s_cand_gid[kMaxRanks], s_cand_slot[kMaxRanks];
  // rotary: the layer's previous-slot entries and those slots' occupants, the window of slots from
  // the hand (occupant, previous occupant)
  constexpr int kWin = 2 * kMaxRanks + 1;
  __shared__ int s_ps_e[256], s_ps_gid[256];
  __shared__ int s_win_gid[kWin], s_win_prior[kWin];
  __shared__ int s_hand;
  __shared__ unsigned long long s_ckey[kFWarps][kMaxRanks];  // each warp's smallest candidate keys
  __shared__ int s_cslot[kFWarps][kMaxRanks];
  // router-guided: the layer's logits and ranks, the refreshed keys of its residents that the step
  // does not use (~0 otherwise), their nev smallest, and the candidates' keys
  __shared__ float s_z[256];
  __shared__ int s_rank[256];
  __shared__ unsigned long long s_lkey[256];
  __shared__ unsigned long long s_lsel[kMaxRanks];
  __shared__ unsigned long long s_cand_key[kMaxRanks];
  const int k = a.k, E = a.E;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  if (warp == 0) {
    int my_i;
    float my_g;
    warp_topk(a.z + (int64_t)l * E, E, k, a.renorm, lane, my_i, my_g);
    if (lane < k && (my_i < 0 || my_i >= E)) {
      atomicOr(a.err, FERR_BAD_ROUTE);
      my_i = lane;  // keep the step well-defined; the host reports the error
    }
    // needed ids in ascending order: each id's position is the count of smaller ids (all distinct)
    const int gid = l * E + my_i;
    int pos = 0;
    for (int t = 0; t < k; t++) {
      const int o = __shfl_sync(kFull, gid, t);
      pos += (lane < k && o < gid) ? 1 : 0;
    }
    if (lane < k) {
      s_idx[lane] = my_i;
      s_gate[lane] = my_g;
      s_need[pos] = gid;
    }
  } else {
    for (int e = threadIdx.x - 32; e < E; e += blockDim.x - 32) s_slot_e[e] = a.slot_of[l * E + e];
    if (threadIdx.x == 32) {
      s_nused = *a.n_used;
      s_trace_base = *(volatile unsigned long long*)a.trace_n;
    }
    if (a.policy == 1) {
      // occupant of slot s: the low 32 bits of its key, or -1 when empty (key all ones)
      auto occupant = [&](int64_t sl) {
        const unsigned long long key = __ldcg(a.slot_key + sl);
        return key == ~0ull ? -1 : (int)(uint32_t)(key & 0xffffffffull);
      };
      for (int e = threadIdx.x - 32; e < E; e += blockDim.x - 32) {
        const int ps = a.prior_slot_of[l * E + e];
        s_ps_e[e] = ps;
        s_ps_gid[e] = ps >= 0 ? occupant(ps) : -1;
      }
      if (warp == 3) {
        const int h0 = *a.hand;
        if (lane == 0) s_hand = h0;
        const int nw = 2 * k + 1 < a.cap ? 2 * k + 1 : (int)a.cap;
        for (int j = lane; j < nw; j += 32) {
          const int64_t sl = (h0 + j) % a.cap;
          s_win_gid[j] = occupant(sl);
          s_win_prior[j] = a.prior[sl];
        }
      }
    }
    if (warp == 2 && lane < k) {
      const int nc = (int)__ldcg(a.cand + kMaxRanks);
      if (lane == 0) s_ncand = nc;
      if (lane < nc) {
        const unsigned long long key = __ldcg(a.cand + lane);
        const int g = slot_key_gid(key, a.policy);
        const bool ok = g >= 0 && g < a.L * E;  // a free slot's key (~0) names no expert
        s_cand_key[lane] = ok ? key : ~0ull;
        s_cand_gid[lane] = ok ? g : -1;
        s_cand_slot[lane] = ok ? a.slot_of[g] : -1;
      }
    }
    if (a.policy == 2)
      for (int e = threadIdx.x - 32; e < E; e += blockDim.x - 32) s_z[e] = __ldcg(a.z + (int64_t)l * E + e);
  }
  __syncthreads();
  if (threadIdx.x < k) {
    const int sl = s_slot_e[s_need[threadIdx.x] - l * E];
    s_slot[threadIdx.x] = sl;
    s_miss[threadIdx.x] = sl < 0;
    s_evict[threadIdx.x] = -1;
  }
  __syncthreads();
  if (a.policy == 1) {
    if (threadIdx.x == 0) rotary_place(a, l, clock, k, E, s_need, s_miss, s_slot, s_evict, s_ps_e, s_ps_gid, s_win_gid,
                                       s_win_prior, s_hand, s_nused, pend);
    __syncthreads();
  }
  if (a.policy == 2) {
    // Refresh the layer's ranks from this routing (rank = logits that beat the expert's, ties to the
    // lower id, in the top-k's order), and the keys of its residents this step does not use; the
    // used ones get their keys below, with this step's clock.
    for (int e = threadIdx.x; e < E; e += blockDim.x) {
      const uint32_t ke = ord_key(s_z[e]);
      int rank = 0;
      for (int j = 0; j < E; j++) {
        const uint32_t kj = ord_key(s_z[j]);
        rank += (kj > ke || (kj == ke && j < e)) ? 1 : 0;
      }
      s_rank[e] = rank;
      a.rank[l * E + e] = rank;
      const int g = l * E + e;
      const int sl = s_slot_e[e];
      bool used = false;
      for (int t = 0; t < k; t++) used |= s_need[t] == g;
      unsigned long long lk = ~0ull;
      if (sl >= 0 && !used) {
        lk = guided_key(E, rank, guided_key_last_use(__ldcg(a.slot_key + sl)), g);
        a.slot_key[sl] = lk;
      }
      s_lkey[e] = lk;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0 && (a.policy == 0 || a.policy == 2)) {
    // misses in ascending id take free slots [n_used, cap) first
    int n_used = s_nused;
    int nev = 0;
    for (int t = 0; t < k; t++) {
      if (s_slot[t] >= 0) continue;
      if (n_used < a.cap)
        s_slot[t] = n_used++;
      else
        nev++;
    }
    if (n_used != s_nused) *a.n_used = n_used;
    s_nev = nev;
    if (a.policy == 2) s_nev_found = 0;  // the guided merge below decides
    // Victims: the nev smallest slot keys (last use, id) among slots that hold no expert of this
    // step (every slot is occupied when eviction is needed). They are among the k smallest keys
    // of the pool (at most k - nev of those belong to this step's hits), which phase C of the
    // previous layer-step left in a.cand. s_nev_found < nev sends the phase to the full scan.
    if (a.policy == 0) {
      int j = 0;
      for (int c = 0; c < s_ncand && j < nev; c++) {
        const int g = s_cand_gid[c];
        if (g < 0) break;  // ascending keys: only free slots' keys follow
        bool needed = false;
        for (int t = 0; t < k; t++) needed |= (s_need[t] == g);
        if (needed) continue;
        s_vgid[j] = g;
        s_vslot[j] = s_cand_slot[c];
        j++;
      }
      s_nev_found = j;
    }
  }
  __syncthreads();
  const int nev = (a.policy == 0 || a.policy == 2) ? s_nev : 0;
  if (a.policy == 2 && nev > 0) {
    // Victims: the nev smallest keys among residents this step does not use. Only this layer's keys
    // changed since phase C of the previous layer-step left the pool's k smallest keys in a.cand,
    // so the candidates of other layers, ascending, are still the smallest keys of other layers;
    // merge them with the nev smallest refreshed keys of this layer. Running out of candidates
    // before nev victims sends the phase to the full scan.
    if (warp == 0) {
      unsigned long long lk[8];
#pragma unroll
      for (int q = 0; q < 8; q++) {
        const int e = q * 32 + lane;
        lk[q] = e < E ? s_lkey[e] : ~0ull;
      }
      for (int j = 0; j < nev; j++) {
        unsigned long long best = ~0ull;
        int bq = 0;
#pragma unroll
        for (int q = 0; q < 8; q++)
          if (lk[q] < best) {
            best = lk[q];
            bq = q;
          }
        const unsigned long long wmin = shfl_min_u64(best);
        const unsigned win = __ballot_sync(kFull, best == wmin && wmin != ~0ull);
        if (win && lane == __ffs(win) - 1) {
#pragma unroll
          for (int q = 0; q < 8; q++)
            if (q == bq) lk[q] = ~0ull;
        }
        if (lane == 0) s_lsel[j] = wmin;
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int c = 0, li = 0, j = 0;
      for (; j < nev; j++) {
        while (c < s_ncand && s_cand_gid[c] >= 0 && s_cand_gid[c] / E == l) c++;  // this layer's are stale
        if (c >= s_ncand || s_cand_gid[c] < 0) break;  // other layers' next key unknown: full scan
        const unsigned long long ck = s_cand_key[c];
        const unsigned long long lk = s_lsel[li];
        if (lk < ck) {
          const int g = slot_key_gid(lk, 2);
          s_vgid[j] = g;
          s_vslot[j] = s_slot_e[g - l * E];
          li++;
        } else {
          s_vgid[j] = s_cand_gid[c];
          s_vslot[j] = s_cand_slot[c];
          c++;
        }
      }
      s_nev_found = j;
    }
    __syncthreads();
  }
  if (nev > 0 && s_nev_found < nev) {  // (LRU and router-guided: nev is 0 under the rotary policy)
    // Full scan: each warp finds the nev smallest of its slots, warp 0 takes the nev smallest of
    // those candidates.
    for (int j = 0; j < nev; j++) {
      unsigned long long best = ~0ull;
      int bslot = -1;
      for (int64_t sl = threadIdx.x; sl < a.cap; sl += blockDim.x) {
        bool skip = false;
        for (int t = 0; t < k; t++) skip |= (s_slot[t] == sl);  // hits are pinned; misses not yet placed
        for (int t = 0; t < j; t++) skip |= (s_cslot[warp][t] == sl);
        if (skip) continue;
        const unsigned long long key = a.slot_key[sl];
        if (key < best) {
          best = key;
          bslot = (int)sl;
        }
      }
      const unsigned long long wmin = shfl_min_u64(best);
      const unsigned win = __ballot_sync(kFull, best == wmin);
      const int leader = __ffs(win) - 1;
      const int wslot = __shfl_sync(kFull, bslot, leader);
      if (lane == 0) {
        s_ckey[warp][j] = wmin;
        s_cslot[warp][j] = wmin == ~0ull ? -1 : wslot;
      }
      __syncwarp();
    }
    __syncthreads();
    if (warp == 0) {
      const int nc = kFWarps * nev;  // <= 128 candidates, 4 per lane
      unsigned long long ck[4];
      int cs[4];
#pragma unroll
      for (int q = 0; q < 4; q++) {
        const int c = q * 32 + lane;
        ck[q] = c < nc ? s_ckey[c / nev][c % nev] : ~0ull;
        cs[q] = c < nc ? s_cslot[c / nev][c % nev] : -1;
      }
      for (int j = 0; j < nev; j++) {
        unsigned long long best = ~0ull;
        int bq = 0;
#pragma unroll
        for (int q = 0; q < 4; q++)
          if (ck[q] < best) {
            best = ck[q];
            bq = q;
          }
        const unsigned long long wmin = shfl_min_u64(best);
        const unsigned win = __ballot_sync(kFull, best == wmin && wmin != ~0ull);
        const int leader = win ? __ffs(win) - 1 : 0;
        int vslot = -1;
#pragma unroll
        for (int q = 0; q < 4; q++)
          if (q == bq) vslot = cs[q];
        vslot = __shfl_sync(kFull, vslot, leader);
        if (lane == leader && win) {
#pragma unroll
          for (int q = 0; q < 4; q++)
            if (q == bq) ck[q] = ~0ull;
        }
        if (lane == 0) {
          if (!win) atomicOr(a.err, FERR_NO_VICTIM);
          s_vslot[j] = win ? vslot : -1;
          s_vgid[j] = win ? slot_key_gid(wmin, a.policy) : -1;
        }
      }
    }
    __syncthreads();
  }
  if (threadIdx.x == 0 && (a.policy == 0 || a.policy == 2)) {
    int j = 0;
    unsigned long long hits = 0, misses = 0, evictions = 0;
    for (int t = 0; t < k; t++) {
      const int g = s_need[t];
      if (!s_miss[t]) {
        hits++;
        continue;
      }
      misses++;
      if (s_slot[t] < 0) {  // needs a victim
        const int vs = s_vslot[j];
        const int v = s_vgid[j];
        j++;
        if (vs >= 0) {
          pend.set(v, -1);
          s_slot[t] = vs;
          s_evict[t] = v;
          evictions++;
        }
      }
      if (s_slot[t] >= 0) pend.set(g, s_slot[t]);
    }
    for (int t = 0; t < k; t++) {
      if (s_slot[t] < 0) continue;
      a.slot_key[s_slot[t]] = a.policy == 2
                                  ? guided_key(E, s_rank[s_need[t] - l * E], (uint32_t)clock, s_need[t])
                                  : ((unsigned long long)(uint32_t)clock << 32) | (uint32_t)s_need[t];
    }
    atomicAdd(a.stats + STAT_HITS, hits);
    atomicAdd(a.stats + STAT_MISSES, misses);
    atomicAdd(a.stats + STAT_EVICTIONS, evictions);
    atomicAdd(a.stats + STAT_LAYER_STEPS, 1ull);
    a.cand[kMaxRanks] = 0ull;  // the keys changed: phase C finds new candidates if the pool is full
  }
  __syncthreads();
  if (threadIdx.x < k) {
    const int t = threadIdx.x;
    const unsigned long long base = s_trace_base;
    if (base + t < (unsigned long long)a.trace_cap) {
      TraceRec rec;
      rec.step = (int32_t)step;
      rec.layer = l;
      rec.expert = s_need[t] - l * E;
      rec.kind = s_miss[t];
      rec.slot = s_slot[t];
      rec.evicted = s_evict[t];
      a.trace[base + t] = rec;
    }
    // plan of rank t
    const int g = l * E + s_idx[t];
    int q = 0;
    while (s_need[q] != g) q++;
    a.plan_slot[po + t] = s_slot[q] < 0 ? 0 : s_slot[q];
    a.plan_gid[po + t] = g;
    a.plan_miss[po + t] = s_miss[q];
    a.plan_gate[po + t] = s_gate[t];
    a.route_idx[l * k + t] = s_idx[t];
    a.route_gate[l * k + t] = s_gate[t];
  }
  __syncthreads();
  if (threadIdx.x == 0) *a.trace_n = s_trace_base + k;
}

// Copy n bf16 values (scales) from src to dst with 2-byte accesses, one per lane.
__device__ __forceinline__ void copy_scales(uint16_t* dst, const uint16_t* src, int n, int lane) {
  for (int j = lane; j < n; j += 32) dst[j] = __ldg(src + j);
}

template <int WD>
__device__ __forceinline__ float scale_at(const uint16_t* p, bool from_host) {
  return bf16_bits(from_host ? __ldg(p) : __ldcg(p));
}

// One gate/up row pair of rank r: reads it from `src` (the host tier for a miss, the slot for a
// hit), stores it into `slot` when it came from the host tier, and writes
// u_r[i] = silu(W_g[i] . x) * (W_u[i] . x) with x staged in shared memory.
template <int WD, int CH>
__device__ __forceinline__ void gateup_row(const FusedArgs& a, const uint8_t* src, uint8_t* slot, bool from_host,
                                           const uint8_t* xs, int r, int i, int lane, float* u = nullptr) {
  const int64_t rb = a.lay.row_bytes_gu;
  const int nch = (int)(rb / 16);
  const int G = a.d / 128;
  const int64_t goff = (int64_t)i * 2 * rb;
  uint4 wg[CH], wu[CH];
#pragma unroll
  for (int j = 0; j < CH; j++) {
    const int c = j * 32 + lane;
    if (c < nch) {
      if (from_host) {
        wg[j] = ld_stream(src + goff + (int64_t)c * 16);
        wu[j] = ld_stream(src + goff + rb + (int64_t)c * 16);
      } else {
        wg[j] = ld_cg(src + goff + (int64_t)c * 16);
        wu[j] = ld_cg(src + goff + rb + (int64_t)c * 16);
      }
    } else {
      wg[j] = make_uint4(0, 0, 0, 0);
      wu[j] = make_uint4(0, 0, 0, 0);
    }
  }
  float sg[CH], su[CH];
  if (WD == WD_INT4) {
    const uint16_t* sp = (const uint16_t*)(src + a.lay.gu_scale_off) + (int64_t)i * 2 * G;
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      sg[j] = c < nch ? scale_at<WD>(sp + (c >> 2), from_host) : 0.f;
      su[j] = c < nch ? scale_at<WD>(sp + G + (c >> 2), from_host) : 0.f;
    }
    if (from_host) copy_scales((uint16_t*)(slot + a.lay.gu_scale_off) + (int64_t)i * 2 * G, sp, 2 * G, lane);
  }
  if (from_host) {
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      if (c < nch) {
        st_v4(slot + goff + (int64_t)c * 16, wg[j]);
        st_v4(slot + goff + rb + (int64_t)c * 16, wu[j]);
      }
    }
  }
  float ag = 0.f, au = 0.f;
#pragma unroll
  for (int j = 0; j < CH; j++) {
    const int c = j * 32 + lane;
    if (c < nch) {
      const uint8_t* xc = xs + (int64_t)c * Tr<WD>::xbytes;
      if (WD == WD_INT4) {
        ag = fmaf(sg[j], dot_chunk<WD>(wg[j], xc, 0.f), ag);
        au = fmaf(su[j], dot_chunk<WD>(wu[j], xc, 0.f), au);
      } else {
        ag = dot_chunk<WD>(wg[j], xc, ag);
        au = dot_chunk<WD>(wu[j], xc, au);
      }
    }
  }
  ag = warp_sum(ag);
  au = warp_sum(au);
  if (lane == 0) (u ? u : a.u)[(int64_t)r * a.I + i] = ag / (1.0f + expf(-ag)) * au;
}

// Stage the k u vectors ([k x I] fp32, rank-major) into shared memory, padded by 4 floats per
// 32 so the 16-byte reads of a warp spread over all banks.
__device__ __forceinline__ void stage_u(const FusedArgs& a, float* us, int ipad, const float* u = nullptr) {
  const float4* u4 = reinterpret_cast<const float4*>(u ? u : a.u);
  const int n4 = a.k * a.I / 4;
#pragma unroll 4
  for (int q = threadIdx.x; q < n4; q += blockDim.x) {
    const float4 v = __ldcg(u4 + q);
    const int r = (4 * q) / a.I;
    const int i = 4 * q - r * a.I;
    *reinterpret_cast<float4*>(us + r * ipad + upad(i)) = v;
  }
}

// Phase D (all experts in their slots) for one value of the chunks-per-lane count of a W_d row:
// stages u, then out[o] = sum_r g_r (W_d^(r)[o] . u_r). A warp's first rows are requested before
// the CTA stages u, so the HBM latency overlaps the staging.
// With np > 1 (the lookahead kernel's layer groups) the phase covers layers l .. l + np - 1 at once:
// pslot / pgate hold np plans of kMaxRanks entries, u the np layers' k x I vectors one after the
// other, us room for np staged copies; rows q = m * d + o (layer l + m, output row o) are spread
// over the warps, each computed exactly as with np = 1.
template <int WD, int CHD>
__device__ void down_phase(const FusedArgs& a, float* us, const int* pslot, const float* pgate, int l, int gw,
                           int W, const float* u = nullptr, bool cta_active = true, int np = 1) {
  if (!cta_active) return;  // the same for every thread of the CTA
  constexpr int E = Tr<WD>::epc;
  constexpr int KR = 24 / CHD > 8 ? 8 : (24 / CHD < 1 ? 1 : 24 / CHD);
  const int lane = threadIdx.x & 31;
  const int64_t rb = a.lay.row_bytes_d;
  const int nch = (int)(rb / 16);
  const int G = a.I / 128;
  const int ipad = ipad_of(a.I);
  const int rows = np * a.d;
  uint4 w[KR][CHD];
  float sc[KR][CHD];
  // loads of ranks [r0, r0 + KR) of row q into w / sc (predicated, no break: keeps them in registers)
  auto issue = [&](int q, int r0) {
    const int m = q < rows ? q / a.d : 0;
    const int o = q < rows ? q - m * a.d : a.d;
#pragma unroll
    for (int rr = 0; rr < KR; rr++) {
      const int r = r0 + rr;
      const bool rok = r < a.k && o < a.d;
      const uint8_t* slot = a.pool + (int64_t)pslot[m * kMaxRanks + (r < a.k ? r : 0)] * a.slot_stride;
      const int64_t roff = a.lay.d_off + (int64_t)(o < a.d ? o : 0) * rb;
#pragma unroll
      for (int j = 0; j < CHD; j++) {
        const int c = j * 32 + lane;
        w[rr][j] = (rok && c < nch) ? ld_cg(slot + roff + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
      }
      if (WD == WD_INT4) {
        const uint16_t* sp = (const uint16_t*)(slot + a.lay.d_scale_off) + (int64_t)(o < a.d ? o : 0) * G;
#pragma unroll
        for (int j = 0; j < CHD; j++) {
          const int c = j * 32 + lane;
          sc[rr][j] = (rok && c < nch) ? scale_at<WD>(sp + (c >> 2), false) : 0.f;
        }
      }
    }
  };
  issue(gw, 0);
  for (int m = 0; m < np; m++)
    stage_u(a, us + (int64_t)m * a.k * ipad, ipad, (u ? u : a.u) + (int64_t)m * a.k * a.I);
  __syncthreads();
  for (int q = gw; q < rows; q += W) {
    const int m = q / a.d;
    const int o = q - m * a.d;
    float acc = 0.f;
    for (int r0 = 0; r0 < a.k; r0 += KR) {
      if (q != gw || r0 != 0) issue(q, r0);
#pragma unroll
      for (int rr = 0; rr < KR; rr++) {
        const int r = r0 + rr;
        if (r >= a.k) continue;
        const float* ur = us + (int64_t)m * a.k * ipad + r * ipad;
        float part = 0.f;
#pragma unroll
        for (int j = 0; j < CHD; j++) {
          const int c = j * 32 + lane;
          if (c < nch) {
            if (WD == WD_INT4)
              part = fmaf(sc[rr][j], dot_chunk_u<WD>(w[rr][j], ur + upad(c * E), 0.f), part);
            else
              part = dot_chunk_u<WD>(w[rr][j], ur + upad(c * E), part);
          }
        }
        acc = fmaf(pgate[m * kMaxRanks + r], part, acc);
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) {
      if (WD == WD_FP32)
        reinterpret_cast<float*>(a.out)[(int64_t)(l + m) * a.d + o] = acc;
      else
        reinterpret_cast<__nv_bfloat16*>(a.out)[(int64_t)(l + m) * a.d + o] = __float2bfloat16_rn(acc);
    }
  }
}

template <int WD, int CH>
__global__ void __launch_bounds__(kFThreads, 2) k_fused(const __grid_constant__ FusedArgs a) {
  extern __shared__ uint4 smem4[];
  __shared__ int p_slot[kMaxRanks], p_gid[kMaxRanks], p_miss[kMaxRanks];
  __shared__ float p_gate[kMaxRanks];
  __shared__ int p_mr[kMaxRanks], p_hr[kMaxRanks], p_nm, p_nh;  // miss / hit ranks of this layer-step
  __shared__ PendingTable pend;                                    // CTA 0: the step's held-back table writes
  const int asize = WD == WD_FP32 ? 4 : 2;
  const int xbytes = a.d * asize;
  uint8_t* xs = reinterpret_cast<uint8_t*>(smem4);
  float* us = reinterpret_cast<float*>(xs + ((xbytes + 15) & ~15));
  const int lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kFWarps + (threadIdx.x >> 5);
  const int W = gridDim.x * kFWarps;
  const int64_t step = *(volatile int64_t*)a.step;
  const int nchr = xbytes / 16;  // router rows: fp32 with fp32 weights, else bf16 (same bytes as h)
  const int ipad = ipad_of(a.I);
  int chd_need = (int)((a.lay.row_bytes_d / 16 + 31) / 32);
  unsigned nbar = 0;  // grid barriers passed in this launch
  if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[a.L * 4] = gtimer();

  for (int l = a.l_begin; l < a.l_end; l++) {
    const int clock = (int)(step * a.L + l + 1);  // 0 is older than every step (preloaded experts)
    // ---- phase R: router logits. A warp's row loads (8 chunks per lane at a time) are issued
    // before the CTA stages h, so their latency overlaps the staging.
    {
      constexpr int RG = 8;
      const bool has_row = gw < a.E;  // at most one row per warp (the grid has >= E warps)
      const uint8_t* row = a.routers + ((int64_t)l * a.E + (has_row ? gw : 0)) * xbytes;
      uint4 rw[RG];
#pragma unroll
      for (int j = 0; j < RG; j++) {
        const int c = j * 32 + lane;
        rw[j] = (has_row && c < nchr) ? ld_stream(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
      }
      stage16(reinterpret_cast<uint4*>(xs), (const uint8_t*)a.hidden + (int64_t)l * xbytes, xbytes, threadIdx.x,
              blockDim.x);
      __syncthreads();
      if (has_row) {
        float acc = 0.f;
        for (int c0 = 0; c0 < nchr; c0 += 32 * RG) {
          if (c0 > 0) {
#pragma unroll
            for (int j = 0; j < RG; j++) {
              const int c = c0 + j * 32 + lane;
              rw[j] = c < nchr ? ld_stream(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
            }
          }
#pragma unroll
          for (int j = 0; j < RG; j++) {
            const int c = c0 + j * 32 + lane;
            if (c < nchr) {
              if (WD == WD_FP32)
                acc = dot_chunk<WD_FP32>(rw[j], xs + (int64_t)c * 16, acc);
              else
                acc = dot_chunk<WD_BF16>(rw[j], xs + (int64_t)c * 16, acc);
            }
          }
        }
        acc = warp_sum(acc);
        if (lane == 0) a.z[(int64_t)l * a.E + gw] = acc;
      }
    }
    if (!grid_sync(a, nbar)) return;
    if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[l * 4 + 0] = gtimer();
    // ---- selection, in every CTA: the same top-k as phase S computes, and hit or miss from the
    // lookup table as it was before this step (phase S holds its table writes back until phase D,
    // and a selected expert that is resident keeps its slot). Hits need nothing else from S.
    if (threadIdx.x < 32) {
      int my_i;
      float my_g;
      warp_topk(a.z + (int64_t)l * a.E, a.E, a.k, a.renorm, lane, my_i, my_g);
      if (lane < a.k) {
        if (my_i < 0 || my_i >= a.E) my_i = lane;  // as phase S does (it reports the error)
        const int gid = l * a.E + my_i;
        const int sl = __ldcg(a.slot_of + gid);
        p_gid[lane] = gid;
        p_gate[lane] = my_g;
        p_miss[lane] = sl < 0;
        p_slot[lane] = sl < 0 ? 0 : sl;  // a miss's slot comes with CTA 0's plan
      }
    }
    // ---- phase S: the lookup-table step (CTA 0), then its plan is published to the miss CTAs
    if (blockIdx.x == 0) {
      if (threadIdx.x == 0) pend.n = 0;
      select_and_lookup(a, l, clock, step, pend);
      __syncthreads();
      if (threadIdx.x == 0) {
        __threadfence();
        asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(a.plan_flag), "r"((unsigned)clock) : "memory");
        if (a.phase_ts) a.phase_ts[l * 4 + 1] = gtimer();
      }
    }
    __syncthreads();
    // ---- phase C: gate-up rows; miss CTAs stream the missed experts into their slots
    if (threadIdx.x == 0) {
      int nm = 0, nh = 0;
      for (int r = 0; r < a.k; r++) {
        if (p_miss[r])
          p_mr[nm++] = r;
        else
          p_hr[nh++] = r;
      }
      p_nm = nm;
      p_nh = nh;
    }
    __syncthreads();
    const int nm = p_nm, nh = p_nh;
    // Warm the host-link address translations of every missed expert before streaming it: one
    // L2 prefetch per page-sized stride, issued by every thread of the grid at once. Without it
    // the streaming warps meet each page's translation miss one after another as they advance
    // through the expert, and the link idles while the translations resolve.
    if (nm > 0 && a.touch_shift > 0) {
      const int64_t pages = (a.lay.total + (1 << a.touch_shift) - 1) >> a.touch_shift;
      const int64_t gt0 = (int64_t)blockIdx.x * kFThreads + threadIdx.x;
      const int64_t GT = (int64_t)gridDim.x * kFThreads;
      for (int64_t q = gt0; q < (int64_t)nm * pages; q += GT) {
        const int m = (int)(q / pages);
        const uint8_t* pa = a.arena + (int64_t)p_gid[p_mr[m]] * a.slot_stride + ((q - (int64_t)m * pages) << a.touch_shift);
        asm volatile("prefetch.global.L2 [%0];" ::"l"(pa));
      }
    }
    // CTA 0 leads phase S and computes no hit rows; with a full pool that can evict it then finds
    // the next layer-step's victim candidates.
    if (blockIdx.x == 0 && a.may_evict && __ldcg(a.n_used) >= a.cap) find_victim_candidates(a);
    const int mctas = nm > 0 ? (a.miss_ctas < (int)gridDim.x - 2 ? a.miss_ctas : (int)gridDim.x - 2) : 0;
    const bool miss_cta = (int)blockIdx.x >= (int)gridDim.x - mctas;  // the last CTAs
    bool plan_ok = true;
    if (miss_cta) {
      // the misses' slots: wait (bounded) for CTA 0's plan of this layer-step
      __shared__ int s_plan_ok;
      if (threadIdx.x == 0) {
        int ok = 1;
        if ((int)(ld_acquire_u32(a.plan_flag) - (unsigned)clock) < 0) {
          const uint64_t t0 = gtimer();
          while ((int)(ld_acquire_u32(a.plan_flag) - (unsigned)clock) < 0) {
            if (*(volatile int*)a.err & FERR_FATAL) {
              ok = 0;
              break;
            }
            if (gtimer() - t0 > a.barrier_timeout_ns) {
              atomicOr(a.err, FERR_BARRIER_TIMEOUT);
              ok = 0;
              break;
            }
            __nanosleep(20);
          }
        }
        s_plan_ok = ok;
      }
      __syncthreads();
      plan_ok = s_plan_ok != 0;
      if (plan_ok && threadIdx.x < a.k && p_miss[threadIdx.x]) p_slot[threadIdx.x] = __ldcg(a.plan_slot + threadIdx.x);
      __syncthreads();
    }
    if (miss_cta && plan_ok) {
      const int mw = ((int)blockIdx.x - ((int)gridDim.x - mctas)) * kFWarps + (threadIdx.x >> 5);
      const int MW = mctas * kFWarps;
      // gate/up rows of every missed expert: host -> slot, and u from the same registers
      for (int p = mw; p < nm * a.I; p += MW) {
        const int r = p_mr[p / a.I];
        const int i = p - (p / a.I) * a.I;
        uint8_t* slot = a.pool + (int64_t)p_slot[r] * a.slot_stride;
        const uint8_t* src = a.arena + (int64_t)p_gid[r] * a.slot_stride;
        gateup_row<WD, CH>(a, src, slot, true, xs, r, i, lane);
      }
      // W_d rows (and int4 scales) of every missed expert: a plain copy host -> slot
      const int64_t dbytes = a.lay.total - a.lay.d_off;  // multiple of 16
      const int64_t nq = dbytes / 16;
      const int mt = ((int)blockIdx.x - ((int)gridDim.x - mctas)) * kFThreads + threadIdx.x;
      const int MT = mctas * kFThreads;
      for (int m = 0; m < nm; m++) {
        const int r = p_mr[m];
        uint8_t* dst = a.pool + (int64_t)p_slot[r] * a.slot_stride + a.lay.d_off;
        const uint8_t* src = a.arena + (int64_t)p_gid[r] * a.slot_stride + a.lay.d_off;
        int64_t q = mt;
        for (; q + 3 * (int64_t)MT < nq; q += 4 * (int64_t)MT) {
          const uint4 v0 = ld_stream(src + q * 16);
          const uint4 v1 = ld_stream(src + (q + MT) * 16);
          const uint4 v2 = ld_stream(src + (q + 2 * (int64_t)MT) * 16);
          const uint4 v3 = ld_stream(src + (q + 3 * (int64_t)MT) * 16);
          st_v4(dst + q * 16, v0);
          st_v4(dst + (q + MT) * 16, v1);
          st_v4(dst + (q + 2 * (int64_t)MT) * 16, v2);
          st_v4(dst + (q + 3 * (int64_t)MT) * 16, v3);
        }
        for (; q < nq; q += MT) st_v4(dst + q * 16, ld_stream(src + q * 16));
      }
    } else if (!miss_cta && blockIdx.x != 0) {
      const int hw = ((int)blockIdx.x - 1) * kFWarps + (threadIdx.x >> 5);
      const int HW = ((int)gridDim.x - mctas - 1) * kFWarps;
      // When this layer-step also streams misses over the host link, phase C leaves HBM mostly
      // idle: bring the hit experts' W_d regions into L2 meanwhile, so phase D reads them from L2.
      // (With every expert a hit the prefetches would compete with the gate/up rows instead.)
      if (nm > 0) {
        const int64_t dbytes = a.lay.total - a.lay.d_off;
        const int64_t nlines = (dbytes + 127) >> 7;
        const int64_t t0 = (int64_t)hw * 32 + lane;
        const int64_t T = (int64_t)HW * 32;
        for (int64_t q = t0; q < (int64_t)nh * nlines; q += T) {
          const int m = (int)(q / nlines);
          const uint8_t* pa = a.pool + (int64_t)p_slot[p_hr[m]] * a.slot_stride + a.lay.d_off + ((q - m * nlines) << 7);
          asm volatile("prefetch.global.L2 [%0];" ::"l"(pa));
        }
      }
      for (int p = hw; p < nh * a.I; p += HW) {
        const int r = p_hr[p / a.I];
        const int i = p - (p / a.I) * a.I;
        uint8_t* slot = a.pool + (int64_t)p_slot[r] * a.slot_stride;
        gateup_row<WD, CH>(a, slot, slot, false, xs, r, i, lane);
      }
    }
    if (!grid_sync(a, nbar)) return;
    if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[l * 4 + 2] = gtimer();
    // CTA 0's plan is visible to every CTA now: the misses' slots; CTA 0 applies the step's table
    // writes (the next reader is the next layer-step, after two more barriers)
    if (threadIdx.x < a.k && p_miss[threadIdx.x]) p_slot[threadIdx.x] = __ldcg(a.plan_slot + threadIdx.x);
    if (blockIdx.x == 0 && threadIdx.x == 0) pend.apply(a);
    __syncthreads();
    // ---- phase D: down rows + combine, every expert read from its slot
    switch (chd_need) {
      case 1: down_phase<WD, 1>(a, us, p_slot, p_gate, l, gw, W); break;
      case 2: down_phase<WD, 2>(a, us, p_slot, p_gate, l, gw, W); break;
      case 3: down_phase<WD, 3>(a, us, p_slot, p_gate, l, gw, W); break;
      case 4: down_phase<WD, 4>(a, us, p_slot, p_gate, l, gw, W); break;
      case 5:
      case 6: down_phase<WD, 6>(a, us, p_slot, p_gate, l, gw, W); break;
      default: down_phase<WD, 8>(a, us, p_slot, p_gate, l, gw, W); break;
    }
    if (!grid_sync(a, nbar)) return;
    if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[l * 4 + 3] = gtimer();
  }
  if (a.l_end == a.L && blockIdx.x == 0 && threadIdx.x == 0) *a.step = step + 1;
}

// Barrier among the worker CTAs (1 .. gridDim.x - 1) of the lookahead kernel, bounded like grid_sync.
// The worker CTAs' arrival counters of the lookahead kernel (every CTA but CTA 0 arrives once per
// layer group, on the counter of the group's parity). worker_arrive: this CTA's threads are done
// with group g's writes (u, slots), then one release-add. worker_wait: thread 0 waits (bounded,
// like grid_sync) until every worker has arrived for group g; false in every thread of the CTA
// once a fatal error flag is set. A CTA arrives for g + 2 only after every worker arrived for g,
// so the parity counter reaches its target for g exactly when all of g's arrivals are in, even
// with CTAs one group apart (a single counter would count g + 1's early arrivals as g's).
__device__ void worker_arrive(const FusedArgs& a, int g) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(a.wbar_count + (g & 1)), "r"(1u) : "memory");
  }
}

__device__ bool worker_wait(const FusedArgs& a, int g) {
  __shared__ int s_abort;
  if (threadIdx.x == 0) {
    const unsigned* cnt = a.wbar_count + (g & 1);
    const unsigned target = a.wbar_base[g & 1] + (unsigned)(g / 2 + 1) * (gridDim.x - 1);
    if ((int)(ld_acquire_u32(cnt) - target) < 0) {
      const uint64_t t0 = gtimer();
      while ((int)(ld_acquire_u32(cnt) - target) < 0) {
        if (*(volatile int*)a.err & FERR_FATAL) break;
        if (gtimer() - t0 > a.barrier_timeout_ns) {
          atomicOr(a.err, FERR_BARRIER_TIMEOUT);
          break;
        }
        __nanosleep(20);
      }
    }
    s_abort = *(volatile int*)a.err & FERR_FATAL;
  }
  __syncthreads();
  return s_abort == 0;
}

// Thread 0 waits (bounded) until the counter p has reached target (wrapping compare); false on a
// timeout (sets FERR_BARRIER_TIMEOUT) or when another CTA has flagged a fatal error.
__device__ bool wait_count(const FusedArgs& a, const unsigned* p, unsigned target) {
  if ((int)(ld_acquire_u32(p) - target) >= 0) return true;
  const uint64_t t0 = gtimer();
  while ((int)(ld_acquire_u32(p) - target) < 0) {
    if (*(volatile int*)a.err & FERR_FATAL) return false;
    if (gtimer() - t0 > a.barrier_timeout_ns) {
      atomicOr(a.err, FERR_BARRIER_TIMEOUT);
      return false;
    }
    __nanosleep(20);
  }
  return true;
}

// Phase R of the lookahead kernels: the router logits of every layer, one router row per warp at
// a time, h_l read through L2; RG chunks of the row and of h_l in flight per lane (the same
// per-lane order of chunks as k_fused, so the logits are bit-identical).
template <int WD>
__device__ void la_router_all(const FusedArgs& a, int gw, int W, int lane) {
  const int xbytes = a.d * (WD == WD_FP32 ? 4 : 2);
  const int nchr = xbytes / 16;
  for (int row = gw; row < a.L * a.E; row += W) {
    constexpr int RG = 8;
    const int l = row / a.E;
    const uint8_t* wr = a.routers + (int64_t)row * xbytes;
    const uint8_t* hl = (const uint8_t*)a.hidden + (int64_t)l * xbytes;
    float acc = 0.f;
    for (int c0 = 0; c0 < nchr; c0 += 32 * RG) {
      uint4 w[RG], h[RG];
#pragma unroll
      for (int j = 0; j < RG; j++) {
        const int c = c0 + j * 32 + lane;
        w[j] = c < nchr ? ld_stream(wr + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
        h[j] = c < nchr ? ld_cg(hl + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int j = 0; j < RG; j++) {
        const int c = c0 + j * 32 + lane;
        if (c < nchr) {
          if (WD == WD_FP32)
            acc = dot_chunk<WD_FP32>(w[j], reinterpret_cast<const uint8_t*>(&h[j]), acc);
          else
            acc = dot_chunk<WD_BF16>(w[j], reinterpret_cast<const uint8_t*>(&h[j]), acc);
        }
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) a.z[row] = acc;
  }
}

// CTA 0 of the lookahead kernels: the lookup steps of layers 0 .. L-1 in order (the same calls,
// clocks, trace and table as the layer-by-layer kernel), layer m's plan going to plan[m][k] and
// plan_flag = its clock. s_ok is a shared-memory flag of the calling CTA.
__device__ void la_lookups(const FusedArgs& a, int64_t step, PendingTable& pend, int& s_ok) {
  const int k = a.k;
  for (int m = 0; m < a.L; m++) {
    const int clock = (int)(step * a.L + m + 1);
    if (threadIdx.x == 0) {
      s_ok = (*(volatile int*)a.err & FERR_FATAL) == 0;
      pend.n = 0;
    }
    __syncthreads();
    if (!s_ok) return;
    select_and_lookup(a, m, clock, step, pend, (int64_t)m * k);
    __syncthreads();
    if (threadIdx.x == 0) {
      pend.apply(a);  // nothing else reads the table in this kernel
      __threadfence();
      asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(a.plan_flag), "r"((unsigned)clock) : "memory");
    }
    __syncthreads();
    if (a.may_evict && __ldcg(a.n_used) >= a.cap) find_victim_candidates(a);
    __syncthreads();
  }
  if (threadIdx.x == 0) *a.step = step + 1;
}

// Exact layer lookahead, batch 1, LRU. One launch per decode step:
//   R   router logits of every layer (row l * E + e per warp, hidden read from global memory), then
//       one grid barrier;
//   CTA 0: the lookup step of layers 0 .. L-1 in order (the same calls, clocks, trace and table as
//       the layer-by-layer kernel), layer m's plan going to plan[m][k] and plan_flag = its clock.
//       Table writes change no slot's bytes: those change only when the miss CTAs stream a miss,
//       so CTA 0 may run any number of layers ahead;
//   workers (CTAs 1 ..): the layers in groups of a.la_group. Per group: wait for its plans, the
//       gate-up rows (the last miss_ctas workers stream the missed experts from the host tier into
//       their slots), an arrival on the workers' counter, then the down rows + combine of a group
//       whose arrivals are all in, on the workers that computed its hits: the same group
//       (unskewed) or the one before (skewed). No barrier follows the down rows: the next group's
//       gate-up rows (and the miss CTAs' streaming of its misses) start beside them. A miss lands
//       while the down rows of the groups before may still read; the host picks the group size
//       and the skew so that LRU never hands a miss the slot of an expert they use.
template <int WD, int CH>
__global__ void __launch_bounds__(kFThreads, 2) k_fused_la(const __grid_constant__ FusedArgs a) {
  extern __shared__ uint4 smem4[];
  // The plans of two groups' layers (a.la_group layers each, 1 or kLaGroupMax), by group parity:
  // group g's down rows may run after group g + 1's gate/up rows have loaded their plan.
  __shared__ int p_slot[2][kLaGroupMax][kMaxRanks], p_gid[2][kLaGroupMax][kMaxRanks];
  __shared__ int p_miss[2][kLaGroupMax][kMaxRanks];
  __shared__ float p_gate[2][kLaGroupMax][kMaxRanks];
  __shared__ int p_mr[2][kLaGroupMax][kMaxRanks], p_hr[2][kLaGroupMax][kMaxRanks];
  __shared__ int p_nm[2][kLaGroupMax], p_nh[2][kLaGroupMax], p_mctas[2];
  __shared__ PendingTable pend;
  __shared__ int s_ok;
  const int asize = WD == WD_FP32 ? 4 : 2;
  const int xbytes = a.d * asize;
  const int xpad = (xbytes + 15) & ~15;
  uint8_t* xs0 = reinterpret_cast<uint8_t*>(smem4);               // [la_group][xpad]
  float* us = reinterpret_cast<float*>(xs0 + a.la_group * xpad);  // [la_group][k x ipad]
  const int lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kFWarps + (threadIdx.x >> 5);
  const int W = gridDim.x * kFWarps;
  const int64_t step = *(volatile int64_t*)a.step;
  const int chd_need = (int)((a.lay.row_bytes_d / 16 + 31) / 32);
  const int k = a.k;
  unsigned nbar = 0;

  la_router_all<WD>(a, gw, W, lane);
  if (!grid_sync(a, nbar)) return;
  if (blockIdx.x == 0) {
    la_lookups(a, step, pend, s_ok);
    return;
  }

  // ---- workers: the layers in groups of P = a.la_group. Each worker CTA arrives once per group
  // on the worker counter after its gate/up rows; the down rows of group g start once every
  // worker has arrived for g. Unskewed (a.la_skew = 0) a CTA runs gate/up(g), arrive, wait for g,
  // down(g); skewed (1) it runs gate/up(g), arrive, wait for g - 1, down(g - 1), so the wait
  // almost never stalls and the CTAs' down rows and gate/up rows interleave in HBM.
  const int wgw = ((int)blockIdx.x - 1) * kFWarps + (threadIdx.x >> 5);
  const int P = a.la_group;
  const int G = (a.L + P - 1) / P;
  const int workers = (int)gridDim.x - 1;
  const int skew = a.la_skew;
  // u of group g: 2 (unskewed) or 4 (skewed) sets of P layers' vectors, in turn. Skewed, a CTA
  // writes u of group g after every worker arrived for g - 2, when a CTA may not yet have staged
  // u of g - 3 for its down rows, hence four.
  const int nu = skew ? 4 : 2;
  for (int g = 0; g < G + skew; g++) {
    if (g < G) {
      const int l0 = g * P;
      const int np = a.L - l0 < P ? a.L - l0 : P;
      const int b = g & 1;
      float* ug = a.u + (int64_t)((g % nu) * P) * k * a.I;
      __syncthreads();  // this CTA's down rows of group g - 2 (plan buffer b) and its gate/up rows of g - 1 (x) are done
      if (threadIdx.x == 0) s_ok = wait_count(a, a.plan_flag, (unsigned)(step * a.L + l0 + np));
      __syncthreads();
      if (!s_ok) return;
      if (threadIdx.x < np * k) {
        const int m = threadIdx.x / k, r = threadIdx.x - m * k;
        const int64_t q = (int64_t)(l0 + m) * k + r;
        p_slot[b][m][r] = __ldcg(a.plan_slot + q);
        p_gid[b][m][r] = __ldcg(a.plan_gid + q);
        p_miss[b][m][r] = __ldcg(a.plan_miss + q);
        p_gate[b][m][r] = __ldcg(a.plan_gate + q);
      }
      for (int m = 0; m < np; m++)
        stage16(reinterpret_cast<uint4*>(xs0 + m * xpad), (const uint8_t*)a.hidden + (int64_t)(l0 + m) * xbytes, xbytes,
                threadIdx.x, blockDim.x);
      __syncthreads();
      if (threadIdx.x == 0) {
        int nm_all = 0;
        for (int m = 0; m < np; m++) {
          int nm = 0, nh = 0;
          for (int r = 0; r < k; r++) {
            if (p_miss[b][m][r])
              p_mr[b][m][nm++] = r;
            else
              p_hr[b][m][nh++] = r;
          }
          p_nm[b][m] = nm;
          p_nh[b][m] = nh;
          nm_all += nm;
        }
        p_mctas[b] = nm_all > 0 ? (a.miss_ctas < workers - 1 ? a.miss_ctas : workers - 1) : 0;
      }
      __syncthreads();
      int nm_all = 0, nh_all = 0;
      for (int m = 0; m < np; m++) {
        nm_all += p_nm[b][m];
        nh_all += p_nh[b][m];
      }
      const int mctas = p_mctas[b];
      const bool miss_cta = (int)blockIdx.x >= (int)gridDim.x - mctas;
      if (nm_all > 0 && a.touch_shift > 0) {
        const int64_t pages = (a.lay.total + (1 << a.touch_shift) - 1) >> a.touch_shift;
        const int64_t gt0 = ((int64_t)blockIdx.x - 1) * kFThreads + threadIdx.x;
        const int64_t GT = (int64_t)workers * kFThreads;
        for (int64_t q = gt0; q < (int64_t)nm_all * pages; q += GT) {
          int mi = (int)(q / pages), m = 0;
          while (mi >= p_nm[b][m]) mi -= p_nm[b][m++];  // the group's misses in layer order
          const uint8_t* pa = a.arena + (int64_t)p_gid[b][m][p_mr[b][m][mi]] * a.slot_stride +
                              ((q - (q / pages) * pages) << a.touch_shift);
          asm volatile("prefetch.global.L2 [%0];" ::"l"(pa));
        }
      }
      if (miss_cta) {
        // A miss's bytes go into a slot whose previous expert no reader may still need: every
        // worker must have arrived for g - 1 (unskewed that wait passed before the down rows of
        // g - 1). The readers left are then the down rows of g - 2 (skewed only) and g - 1 and
        // the gate/up rows of g, i.e. at most 3 P - 1 layer-steps before the miss's own, which
        // LRU keeps from 3 P k slots on (2 P k unskewed); the host checks the cap.
        if (g > 0 && !worker_wait(a, g - 1)) return;
        const int mw = ((int)blockIdx.x - ((int)gridDim.x - mctas)) * kFWarps + (threadIdx.x >> 5);
        const int MW = mctas * kFWarps;
        // gate/up rows of every missed expert of the group, layer by layer: host -> slot, and u
        for (int p = mw; p < nm_all * a.I; p += MW) {
          int mi = p / a.I, m = 0;
          while (mi >= p_nm[b][m]) mi -= p_nm[b][m++];
          const int r = p_mr[b][m][mi];
          const int i = p - (p / a.I) * a.I;
          uint8_t* slot = a.pool + (int64_t)p_slot[b][m][r] * a.slot_stride;
          const uint8_t* src = a.arena + (int64_t)p_gid[b][m][r] * a.slot_stride;
          gateup_row<WD, CH>(a, src, slot, true, xs0 + m * xpad, r, i, lane, ug + (int64_t)m * k * a.I);
        }
        const int64_t dbytes = a.lay.total - a.lay.d_off;
        const int64_t nq = dbytes / 16;
        const int mt = ((int)blockIdx.x - ((int)gridDim.x - mctas)) * kFThreads + threadIdx.x;
        const int MT = mctas * kFThreads;
        for (int m = 0; m < np; m++)
          for (int mi = 0; mi < p_nm[b][m]; mi++) {
            const int r = p_mr[b][m][mi];
            uint8_t* dst = a.pool + (int64_t)p_slot[b][m][r] * a.slot_stride + a.lay.d_off;
            const uint8_t* src = a.arena + (int64_t)p_gid[b][m][r] * a.slot_stride + a.lay.d_off;
            for (int64_t q = mt; q < nq; q += MT) st_v4(dst + q * 16, ld_stream(src + q * 16));
          }
      } else {
        const int hw = wgw;
        const int HW = (workers - mctas) * kFWarps;
        for (int p = hw; p < nh_all * a.I; p += HW) {
          int hi = p / a.I, m = 0;
          while (hi >= p_nh[b][m]) hi -= p_nh[b][m++];
          const int r = p_hr[b][m][hi];
          const int i = p - (p / a.I) * a.I;
          uint8_t* slot = a.pool + (int64_t)p_slot[b][m][r] * a.slot_stride;
          gateup_row<WD, CH>(a, slot, slot, false, xs0 + m * xpad, r, i, lane, ug + (int64_t)m * k * a.I);
        }
        // In a group that streams misses the hit workers wait for the miss CTAs before the
        // group's down rows: done with its gate/up rows, a warp requests into L2 the W_d rows of
        // the hit experts that its down rows will read, and those rows then start from L2. (With
        // every expert a hit the requests would only compete with the last gate/up rows: measured
        // 0.59 -> 0.57 of HBM peak resident, while the capped int4 stack gained 18%.)
        if (nm_all > 0) {
          const int64_t rbd = a.lay.row_bytes_d;
          const int nl = (int)((rbd + 127) >> 7);
          for (int q = wgw; q < np * a.d; q += HW) {
            const int m = q / a.d, o = q - m * a.d;
            for (int t = lane; t < p_nh[b][m] * nl; t += 32) {
              const int r = p_hr[b][m][t / nl];
              const uint8_t* pa = a.pool + (int64_t)p_slot[b][m][r] * a.slot_stride + a.lay.d_off +
                                  (int64_t)o * rbd + ((int64_t)(t % nl) << 7);
              asm volatile("prefetch.global.L2 [%0];" ::"l"(pa));
            }
          }
        }
      }
      worker_arrive(a, g);
    }
    // Down rows + combine of group dg on the CTAs that computed its hits: its miss CTAs go
    // straight on to the next group's misses, so the host link stays busy.
    const int dg = g - skew;
    if (dg < 0) continue;
    if (!worker_wait(a, dg)) return;
    const int db = dg & 1;
    const int dl0 = dg * P;
    const int dnp = a.L - dl0 < P ? a.L - dl0 : P;
    const int HWW = (workers - p_mctas[db]) * kFWarps;
    const bool dact = (int)blockIdx.x < (int)gridDim.x - p_mctas[db];
    const int* ps = &p_slot[db][0][0];
    const float* pg = &p_gate[db][0][0];
    const float* ud = a.u + (int64_t)((dg % nu) * P) * k * a.I;
    switch (chd_need) {
      case 1: down_phase<WD, 1>(a, us, ps, pg, dl0, wgw, HWW, ud, dact, dnp); break;
      case 2: down_phase<WD, 2>(a, us, ps, pg, dl0, wgw, HWW, ud, dact, dnp); break;
      case 3: down_phase<WD, 3>(a, us, ps, pg, dl0, wgw, HWW, ud, dact, dnp); break;
      case 4: down_phase<WD, 4>(a, us, ps, pg, dl0, wgw, HWW, ud, dact, dnp); break;
      case 5:
      case 6: down_phase<WD, 6>(a, us, ps, pg, dl0, wgw, HWW, ud, dact, dnp); break;
      default: down_phase<WD, 8>(a, us, ps, pg, dl0, wgw, HWW, ud, dact, dnp); break;
    }
  }
}

size_t fused_smem(int wdtype, int d, int I, int k) {
  const int xbytes = d * (wdtype == WD_FP32 ? 4 : 2);
  return (size_t)((xbytes + 15) & ~15) + (size_t)k * ipad_of(I) * sizeof(float);
}

template <int WD, int CH>
int grid_of(size_t smem) {
  static int occ = -1;
  static size_t occ_smem = 0;
  if (occ < 0 || occ_smem != smem) {
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(k_fused<WD, CH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    int o = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, k_fused<WD, CH>, kFThreads, smem) != cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    occ = o;
    occ_smem = smem;
  }
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = sms * (occ < 2 ? occ : 2);
  return grid * kFWarps >= 256 ? grid : 0;  // phase R gives each expert row its own warp
}

template <int WD, int CH>
cudaError_t run_fused(const FusedArgs& a, int grid, cudaStream_t s) {
  const size_t smem = fused_smem(a.wdtype, a.d, a.I, a.k);
  void* params[] = {(void*)&a};
  return cudaLaunchCooperativeKernel((const void*)k_fused<WD, CH>, dim3(grid), dim3(kFThreads), params, smem, s);
}

int pick_ch_f(int64_t rb) {
  const int need = (int)((rb / 16 + 31) / 32);
  if (need <= 1) return 1;
  if (need <= 2) return 2;
  if (need <= 4) return 4;
  if (need <= 8) return 8;
  if (need <= 16) return 16;
  return -1;
}

}  // namespace

#define MOE_F_DISPATCH(FN, WDV, CHV, ...)                          \
  do {                                                             \
    switch (WDV) {                                                 \
      case WD_FP32:                                                \
        switch (CHV) {                                             \
          case 1: return FN<WD_FP32, 1>(__VA_ARGS__);              \
          case 2: return FN<WD_FP32, 2>(__VA_ARGS__);              \
          case 4: return FN<WD_FP32, 4>(__VA_ARGS__);              \
          case 8: return FN<WD_FP32, 8>(__VA_ARGS__);              \
        }                                                          \
        break;                                                     \
      case WD_BF16:                                                \
        switch (CHV) {                                             \
          case 1: return FN<WD_BF16, 1>(__VA_ARGS__);              \
          case 2: return FN<WD_BF16, 2>(__VA_ARGS__);              \
          case 4: return FN<WD_BF16, 4>(__VA_ARGS__);              \
          case 8: return FN<WD_BF16, 8>(__VA_ARGS__);              \
          case 16: return FN<WD_BF16, 16>(__VA_ARGS__);            \
        }                                                          \
        break;                                                     \
      case WD_INT4:                                                \
        switch (CHV) {                                             \
          case 1: return FN<WD_INT4, 1>(__VA_ARGS__);              \
          case 2: return FN<WD_INT4, 2>(__VA_ARGS__);              \
          case 4: return FN<WD_INT4, 4>(__VA_ARGS__);              \
          case 8: return FN<WD_INT4, 8>(__VA_ARGS__);              \
        }                                                          \
        break;                                                     \
    }                                                              \
  } while (0)

template <int WD, int CH>
int grid_of_la(size_t smem) {
  static int occ = -1;
  static size_t occ_smem = 0;
  if (occ < 0 || occ_smem != smem) {
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(k_fused_la<WD, CH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    int o = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, k_fused_la<WD, CH>, kFThreads, smem) != cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    occ = o;
    occ_smem = smem;
  }
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = sms * (occ < 2 ? occ : 2);
  return grid >= 3 ? grid : 0;  // CTA 0 and at least two workers
}

// The lookahead kernel stages the inputs and u vectors of a whole layer group.
size_t fused_la_smem(int wdtype, int d, int I, int k, int group) {
  return (size_t)group * fused_smem(wdtype, d, I, k);
}

template <int WD, int CH>
cudaError_t run_fused_la(const FusedArgs& a, int grid, cudaStream_t s) {
  const size_t smem = fused_la_smem(a.wdtype, a.d, a.I, a.k, a.la_group);
  void* params[] = {(void*)&a};
  return cudaLaunchCooperativeKernel((const void*)k_fused_la<WD, CH>, dim3(grid), dim3(kFThreads), params, smem, s);
}

int fused_grid(int wdtype, int d, int I, int k) {
  const BlobLayout lay = make_layout(wdtype, d, I);
  const int ch = pick_ch_f(lay.row_bytes_gu);
  const size_t smem = fused_smem(wdtype, d, I, k);
  if (smem > 200 * 1024) return 0;
  MOE_F_DISPATCH(grid_of, wdtype, ch, smem);
  return 0;
}

cudaError_t launch_fused(const FusedArgs& a, int grid, cudaStream_t s) {
  const int ch = pick_ch_f(a.lay.row_bytes_gu);
  MOE_F_DISPATCH(run_fused, a.wdtype, ch, a, grid, s);
  return cudaErrorInvalidValue;
}

int fused_la_grid(int wdtype, int d, int I, int k, int group) {
  const BlobLayout lay = make_layout(wdtype, d, I);
  const int ch = pick_ch_f(lay.row_bytes_gu);
  const size_t smem = fused_la_smem(wdtype, d, I, k, group);
  if (smem > 200 * 1024) return 0;
  MOE_F_DISPATCH(grid_of_la, wdtype, ch, smem);
  return 0;
}

cudaError_t launch_fused_la(const FusedArgs& a, int grid, cudaStream_t s) {
  const int ch = pick_ch_f(a.lay.row_bytes_gu);
  MOE_F_DISPATCH(run_fused_la, a.wdtype, ch, a, grid, s);
  return cudaErrorInvalidValue;
}

}  // namespace moe
