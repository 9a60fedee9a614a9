// Batched device-driven decode step (sm_103a): B sequences decode together, one cooperative
// persistent kernel per step over all layers.
//
// Per layer, six phases separated by grid barriers:
//   R  router logits z[b][e] = W_r[e] . h_b. A warp holds one router row in registers and applies
//      it to a block of 8 sequences;
//   T  per sequence b (one warp each): top k with ties to the lower id, and the gates. Pair
//      p = b * k + r is rank r of sequence b;
//   S  CTA 0: the needed experts are the union of all pairs' experts, ascending. One step of the
//      lookup table for that set: hits keep their slot, misses (ascending id) take the lowest
//      free slots, then the residents that no pair needs, smallest (last use, id) first (a bitonic
//      sort of the slot keys in shared memory). It writes one trace record per needed expert, and
//      the plan: the needed experts (misses first, then hits) with their slots and, per expert,
//      the ascending list of pairs routed to it;
//   C  grouped gate-up: a work item is (needed expert, block of rows). The CTA stages the
//      activations of the expert's pairs in shared memory, and each warp reads a row pair once
//      and applies it to every staged pair: u_p[i] = silu(W_g[i] . h_b) * (W_u[i] . h_b). A
//      missed expert's item reads its rows from the page-locked host tier over NVLink-C2C,
//      stores them into the expert's slot and uses them from registers, and copies its share of
//      the expert's W_d region into the slot. CTAs take items from a global counter, the missed
//      experts' items first: while misses remain every CTA streams the host tier (many misses per
//      layer-step need all the requests in flight the grid can issue), and the hit items fill in
//      behind them;
//   D  grouped down projection: a work item is (needed expert, block of W_d rows); the CTA stages
//      u of the expert's pairs and each warp applies its rows to all of them, y_p = W_d u_p.
//      Items again come from a global counter (experts with many pairs take longer);
//   E  combine per sequence in rank order: out[b] = sum_r g_{b,r} y_{b*k+r}.
//
// Each expert is read from memory once per layer-step however many pairs it serves. All CTAs are
// co-resident; every barrier wait is bounded and sets an error flag on expiry.
#include <cuda_bf16.h>
#include <math.h>

#include <algorithm>

#include "dev.cuh"
#include "fused.cuh"
#include "grid.cuh"
#include "tc.cuh"
#include "topk.cuh"

namespace moe {
namespace {

using namespace dev;

constexpr int kBWarps = 8;
constexpr int kBThreads = kBWarps * 32;
constexpr int kMaxPairs = kMaxBatch * kMaxRanks;
constexpr int kRowsGU = 64;   // gate/up row pairs per work item
constexpr int kRowsD = 128;   // W_d rows per work item
constexpr int kTGMax = 16;    // pairs staged per group

int tg_of(int wdtype, int d, int I) {
  const int xpad = (d * (wdtype == WD_FP32 ? 4 : 2) + 15) & ~15;
  const int per = std::max(xpad, ipad_of(I) * 4);
  return std::max(1, std::min(kTGMax, (96 * 1024) / per));
}

int sort_n_of(int64_t cap, int64_t n_gid) {
  if (cap >= n_gid) return 0;  // never evicts
  int n = 1;
  while (n < cap) n <<= 1;
  return n;
}

size_t batched_smem(int wdtype, int d, int I, int64_t cap, int64_t n_gid) {
  const int xpad = (d * (wdtype == WD_FP32 ? 4 : 2) + 15) & ~15;
  const size_t per = (size_t)std::max(xpad, ipad_of(I) * 4);
  return std::max((size_t)tg_of(wdtype, d, I) * per, (size_t)sort_n_of(cap, n_gid) * sizeof(unsigned long long));
}

// ---- phase R: a CTA work item is (block of up to rtb sequences, block of 8 router rows). The
// CTA stages the sequences' activations in shared memory; warp w holds row 8 * eb + w in
// registers (its loads are issued before the staging, so their latency overlaps it) and dots it
// with every staged activation vector.
template <int WDR>
__device__ __forceinline__ void router_block(const BatchArgs& a, int l, int tb, int eb, int rtb, uint8_t* xs) {
  constexpr int RG = 8;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int xbytes = a.d * (WDR == WD_FP32 ? 4 : 2);
  const int xpad = (xbytes + 15) & ~15;
  const int nchr = xbytes / 16;
  const int e = eb * kBWarps + warp;
  const bool has_row = e < a.E;
  const uint8_t* row = a.routers + ((int64_t)l * a.E + (has_row ? e : 0)) * xbytes;
  const int b0 = tb * rtb;
  const int nt = a.B - b0 < rtb ? a.B - b0 : rtb;
  uint4 rw[RG];
#pragma unroll
  for (int j = 0; j < RG; j++) {
    const int c = j * 32 + lane;
    rw[j] = (has_row && c < nchr) ? ld_cg(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
  }
  __syncthreads();  // the previous item's readers are done with xs
  for (int q = threadIdx.x; q < nt * nchr; q += blockDim.x) {
    const int t = q / nchr, c = q - t * nchr;
    const uint4* src = reinterpret_cast<const uint4*>((const uint8_t*)a.hidden + ((int64_t)l * a.B + b0 + t) * xbytes);
    *reinterpret_cast<uint4*>(xs + (int64_t)t * xpad + (int64_t)c * 16) = __ldg(src + c);
  }
  __syncthreads();
  if (!has_row) return;
#pragma unroll 1
  for (int t = 0; t < nt; t++) {
    const uint8_t* x = xs + (int64_t)t * xpad;
    float acc = 0.f;
    for (int c0 = 0; c0 < nchr; c0 += 32 * RG) {
      if (c0 > 0) {  // rows longer than 256 chunks: the next part (L1/L2 hits after the first vector)
#pragma unroll
        for (int j = 0; j < RG; j++) {
          const int c = c0 + j * 32 + lane;
          rw[j] = c < nchr ? ld_cg(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
        }
      }
#pragma unroll
      for (int j = 0; j < RG; j++) {
        opaque(rw[j]);
        const int c = c0 + j * 32 + lane;
        if (c < nchr) acc = dot_chunk<WDR>(rw[j], x + (int64_t)c * 16, acc);
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) a.z[((int64_t)l * a.Bmax + b0 + t) * a.E + e] = acc;
    if (nchr > 32 * RG && t + 1 < nt) {  // back to the row's first part for the next vector
#pragma unroll
      for (int j = 0; j < RG; j++) {
        const int c = j * 32 + lane;
        rw[j] = c < nchr ? ld_cg(row + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
      }
    }
  }
}

// ---- phase S: union of the pairs' experts, one lookup-table step, trace and plan (CTA 0)
// Rotary slot-group step for the misses of a batched layer-step (thread 0 of CTA 0): the rule of
// the batch-1 kernel applied to the union of the batch's experts, misses in ascending id. A miss
// returns to the slot it was last evicted from when that slot holds no expert of the step
// (reverse rotation), else takes the first such slot at or after the hand, which moves past it
// (forward rotation); the occupant is evicted and remembered as the slot's previous occupant, and
// the placed expert stops being anyone's previous occupant. Up to E misses per step, so the slot
// state is read and written in global memory as it goes rather than staged: the occupant of a slot
// is the low half of its key (all ones: empty), and each placement writes its key at once.
// needed(o): o belongs to layer l and has pairs this step (tot[o - l * E] > 0).
__device__ void batched_rotary_place(const BatchArgs& a, int l, int clock, int n, const int* need_e,
                                     const int* miss, const int* tot, int* slot_out, int* evict_out,
                                     int* n_evicted) {
  const int E = a.E;
  const int64_t cap = a.cap;
  auto occupant = [&](int64_t sl) {
    const unsigned long long key = __ldcg(a.slot_key + sl);
    return key == ~0ull ? -1 : (int)(uint32_t)(key & 0xffffffffull);
  };
  auto needed = [&](int o) { return o >= l * E && o < (l + 1) * E && tot[o - l * E] > 0; };
  int hand = *(volatile int32_t*)a.hand;
  int nused = *(volatile int32_t*)a.n_used;
  int evicted = 0;
  for (int q = 0; q < n; q++) {
    if (!miss[q]) continue;
    const int g = l * E + need_e[q];
    int slot = -1, occ = -1;
    int ps = __ldcg(a.prior_slot_of + g);
    if (ps >= 0 && __ldcg(a.prior + ps) != g) ps = -1;  // the inverse entry is stale
    if (ps >= 0) {
      const int o = occupant(ps);
      if (o < 0 || !needed(o)) {
        slot = ps;
        occ = o;
      }
    }
    if (slot < 0) {
      for (int64_t j = 0; j < cap; j++) {
        const int64_t sl = (hand + j) % cap;
        const int o = occupant(sl);
        if (o < 0 || !needed(o)) {
          slot = (int)sl;
          occ = o;
          break;
        }
      }
      if (slot < 0) {
        atomicOr(a.err, FERR_NO_VICTIM);
        slot_out[q] = -1;
        continue;
      }
      hand = (int)((slot + 1) % cap);
    }
    if (occ >= 0) {
      a.slot_of[occ] = -1;
      evicted++;
    } else {
      nused++;
    }
    if (ps >= 0) a.prior[ps] = -1;  // g is placed: no longer a previous occupant
    const int u = __ldcg(a.prior + slot);  // the slot's previous occupant loses its return slot
    if (u >= 0) a.prior_slot_of[u] = -1;
    a.prior[slot] = occ;
    if (occ >= 0) a.prior_slot_of[occ] = slot;
    a.prior_slot_of[g] = -1;
    a.slot_of[g] = slot;
    a.slot_key[slot] = ((unsigned long long)(uint32_t)clock << 32) | (uint32_t)g;
    __threadfence_block();
    slot_out[q] = slot;
    evict_out[q] = occ;
  }
  *a.hand = hand;
  *a.n_used = nused;
  *n_evicted = evicted;
}

__device__ void batched_select(const BatchArgs& a, int l, int clock, int64_t step, unsigned long long* keys) {
  constexpr int kChunks = kMaxPairs / 32;
  __shared__ int s_sel[kMaxPairs];       // expert of pair p
  __shared__ uint8_t s_rank[kMaxPairs];  // rank of pair p among the pairs of its 32-pair chunk with its expert
  __shared__ uint8_t s_hist[kChunks][256];  // pairs per (chunk, expert), then their prefix over chunks
  __shared__ int s_slot_e[256];          // slot of every expert of the layer before the step (-1: not resident)
  __shared__ int s_tot[256];             // pairs per expert
  __shared__ int s_q_of_e[256];          // index of expert e among the needed experts
  __shared__ int s_need[256];            // needed expert ids (within the layer), ascending
  __shared__ int s_slot[256];
  __shared__ int s_miss[256];
  __shared__ int s_mbefore[256];         // misses among needed[0..q)
  __shared__ int s_evict[256];
  __shared__ int s_pos[256];             // plan position of needed q: misses first, then hits
  __shared__ int s_cnt[256];             // pairs per plan position
  __shared__ int s_off[256];
  __shared__ int s_n, s_nm, s_nused0, s_nfree, s_nev, s_nevicted;
  __shared__ unsigned long long s_trace_base;
  __shared__ int s_grank[256];           // router-guided: each expert's best rank over the batch
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int E = a.E, P = a.B * a.k;
  const int nchunks = (P + 31) / 32;
  const bool guided = a.policy == 2;

  // every global read this step needs, issued together
  for (int p = tid; p < P; p += blockDim.x) s_sel[p] = __ldcg(a.sel_e + p);
  for (int e = tid; e < E; e += blockDim.x) {
    s_slot_e[e] = a.slot_of[l * E + e];
    if (guided) s_grank[e] = __ldcg(a.rank_best + e);
  }
  if (tid == 0) {
    s_nused0 = *a.n_used;
    s_trace_base = *(volatile unsigned long long*)a.trace_n;
    s_nevicted = 0;
  }
  for (int i = tid; i < kChunks * 256 / 4; i += blockDim.x) reinterpret_cast<uint32_t*>(s_hist)[i] = 0u;
  __syncthreads();
  // per 32-pair chunk: pairs per expert, and each pair's rank among its chunk's pairs of that expert
  for (int c = warp; c < nchunks; c += kBWarps) {
    const int p = c * 32 + lane;
    const int e = p < P ? s_sel[p] : -1 - lane;  // distinct values for the lanes past the end
    const unsigned m = __match_any_sync(kFull, e);
    if (p < P) {
      s_rank[p] = (uint8_t)__popc(m & ((1u << lane) - 1u));
      if (lane == __ffs(m) - 1) s_hist[c][e] = (uint8_t)__popc(m);
    }
  }
  __syncthreads();
  // per expert: the prefix of its chunk counts (its pairs in earlier chunks), and its total
  for (int e = tid; e < E; e += blockDim.x) {
    int run = 0;
    for (int c = 0; c < nchunks; c++) {
      const int v = s_hist[c][e];
      s_hist[c][e] = (uint8_t)run;
      run += v;
    }
    s_tot[e] = run;
  }
  __syncthreads();
  if (guided) {
    // the layer's ranks from this step's routing; its residents this step does not use get their
    // refreshed keys before the victims are sorted below (the used ones get theirs with this clock)
    for (int e = tid; e < E; e += blockDim.x) {
      a.rank[l * E + e] = s_grank[e];
      const int sl = s_slot_e[e];
      if (sl >= 0 && s_tot[e] == 0)
        a.slot_key[sl] = guided_key(E, s_grank[e], guided_key_last_use(__ldcg(a.slot_key + sl)), l * E + e);
    }
  }
  if (warp == 0) {
    // needed experts (at least one pair) ascending, with their slots; then the misses' ranks
    int base = 0;
    for (int e0 = 0; e0 < E; e0 += 32) {
      const int e = e0 + lane;
      const int tot = e < E ? s_tot[e] : 0;
      const bool f = tot > 0;
      const unsigned m = __ballot_sync(kFull, f);
      if (f) {
        const int q = base + __popc(m & ((1u << lane) - 1u));
        s_need[q] = e;
        s_q_of_e[e] = q;
        s_slot[q] = s_slot_e[e];
        s_miss[q] = s_slot_e[e] < 0;
        s_evict[q] = -1;
        s_cnt[q] = tot;  // by needed index for now
      }
      base += __popc(m);
    }
    const int n = base;
    __syncwarp();
    int nm = 0;
    for (int q0 = 0; q0 < n; q0 += 32) {
      const int q = q0 + lane;
      const bool f = q < n && s_miss[q];
      const unsigned m = __ballot_sync(kFull, f);
      if (q < n) s_mbefore[q] = nm + __popc(m & ((1u << lane) - 1u));
      nm += __popc(m);
    }
    if (lane == 0) {
      const int nfree = (int)(a.cap - s_nused0);
      const int take = nm < nfree ? nm : nfree;
      if (a.policy != 1) *a.n_used = s_nused0 + take;
      s_n = n;
      s_nm = nm;
      s_nfree = nfree;
      s_nev = nm - take;
    }
  }
  __syncthreads();
  const int n = s_n, nm = s_nm, nfree = s_nfree, nev = s_nev;
  if (a.policy == 1) {
    if (tid == 0 && nm > 0) batched_rotary_place(a, l, clock, n, s_need, s_miss, s_tot, s_slot, s_evict, &s_nevicted);
    __syncthreads();
  } else if (nev > 0) {
    // Every slot is occupied. Sort the slot keys (last use << 32 | id) ascending, with the slots
    // of this step's hits pinned at the maximum: the first nev keys are the victims.
    int N2 = 1;
    while (N2 < a.cap) N2 <<= 1;
    for (int s = tid; s < N2; s += blockDim.x) keys[s] = s < a.cap ? a.slot_key[s] : ~0ull;
    __syncthreads();
    for (int q = tid; q < n; q += blockDim.x)
      if (!s_miss[q]) keys[s_slot[q]] = ~0ull;
    __syncthreads();
    for (int size = 2; size <= N2; size <<= 1) {
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        for (int i = tid; i < N2 / 2; i += blockDim.x) {
          const int lo = 2 * i - (i & (stride - 1));
          const int hi = lo + stride;
          const unsigned long long x = keys[lo], y = keys[hi];
          const bool up = (lo & size) == 0;
          if ((x > y) == up) {
            keys[lo] = y;
            keys[hi] = x;
          }
        }
        __syncthreads();
      }
    }
  }
  // place the misses: free slots first, then the victims in ascending key order
  for (int q = tid; q < n; q += blockDim.x) {
    s_pos[q] = s_miss[q] ? s_mbefore[q] : nm + (q - s_mbefore[q]);
    if (!s_miss[q] || a.policy == 1) continue;
    const int m = s_mbefore[q];
    int slot = -1;
    if (m < nfree) {
      slot = s_nused0 + m;
    } else {
      const unsigned long long key = keys[m - nfree];
      if (key == ~0ull) {
        atomicOr(a.err, FERR_NO_VICTIM);
      } else {
        const int v = slot_key_gid(key, a.policy);
        slot = a.slot_of[v];
        s_evict[q] = v;
        atomicAdd(&s_nevicted, 1);
      }
    }
    s_slot[q] = slot;
  }
  __syncthreads();
  for (int q = tid; q < n; q += blockDim.x) {
    if (s_evict[q] >= 0) a.slot_of[s_evict[q]] = -1;
    s_off[s_pos[q]] = s_cnt[q];  // pairs per plan position (scanned below)
  }
  __syncthreads();
  if (warp == 0) {
    // exclusive scan of the pair counts in plan order: 8 consecutive entries per lane
    int v[8], sum = 0;
#pragma unroll
    for (int j = 0; j < 8; j++) {
      const int q = lane * 8 + j;
      v[j] = q < n ? s_off[q] : 0;
      sum += v[j];
    }
    int inc = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(kFull, inc, off);
      if (lane >= off) inc += o;
    }
    __syncwarp();
    int run = inc - sum;
#pragma unroll
    for (int j = 0; j < 8; j++) {
      const int q = lane * 8 + j;
      if (q < n) {
        s_off[q] = run;
        s_cnt[q] = v[j];  // now by plan position
      }
      run += v[j];
    }
  } else {
    const unsigned long long base_rec = s_trace_base;
    for (int q = tid - 32; q < n; q += blockDim.x - 32) {
      const int gid = l * E + s_need[q];
      const int sl = s_slot[q];
      if (s_miss[q] && sl >= 0) a.slot_of[gid] = sl;
      if (sl >= 0)
        a.slot_key[sl] = guided ? guided_key(E, s_grank[s_need[q]], (uint32_t)clock, gid)
                                : ((unsigned long long)(uint32_t)clock << 32) | (uint32_t)gid;
      if (base_rec + q < (unsigned long long)a.trace_cap) {
        TraceRec rec;
        rec.step = (int32_t)step;
        rec.layer = l;
        rec.expert = s_need[q];
        rec.kind = s_miss[q];
        rec.slot = sl;
        rec.evicted = s_evict[q];
        a.trace[base_rec + q] = rec;
      }
    }
  }
  __syncthreads();
  // the plan: pairs grouped by expert in plan order, ascending pair index within an expert
  for (int p = tid; p < P; p += blockDim.x) {
    const int e = s_sel[p];
    const int pos = s_pos[s_q_of_e[e]];
    a.plan_tok[s_off[pos] + s_hist[p >> 5][e] + s_rank[p]] = p;
  }
  for (int q = tid; q < n; q += blockDim.x) {
    const int pos = s_pos[q];
    const int sl = s_slot[q];
    a.plan_slot[pos] = sl < 0 ? 0 : sl;
    a.plan_gid[pos] = l * E + s_need[q];
    a.plan_miss[pos] = s_miss[q];
    a.plan_off[pos] = s_off[pos];
    a.plan_cnt[pos] = s_cnt[pos];
  }
  if (tid == 0) {
    a.plan_n[0] = n;
    a.plan_n[1] = nm;
    a.work[0] = 0u;  // the previous layer's phases C and D are complete (grid barriers since)
    a.work[1] = 0u;
    *a.trace_n = s_trace_base + n;
    atomicAdd(a.stats + STAT_HITS, (unsigned long long)(n - nm));
    atomicAdd(a.stats + STAT_MISSES, (unsigned long long)nm);
    atomicAdd(a.stats + STAT_EVICTIONS, (unsigned long long)s_nevicted);
    atomicAdd(a.stats + STAT_LAYER_STEPS, 1ull);
  }
}

template <int WD>
__device__ __forceinline__ float scale_b(const uint16_t* p, bool from_host) {
  return bf16_bits(from_host ? __ldg(p) : __ldcg(p));
}

// ---- phase C: one gate/up row pair of an expert applied to the tg staged pairs
template <int WD, int CH>
__device__ __forceinline__ void gateup_rows(const BatchArgs& a, const uint8_t* src, uint8_t* slot, bool from_host,
                                            const uint8_t* xs, int xpad, const int* pidx, int tg, int i, int lane) {
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
      sg[j] = c < nch ? scale_b<WD>(sp + (c >> 2), from_host) : 0.f;
      su[j] = c < nch ? scale_b<WD>(sp + G + (c >> 2), from_host) : 0.f;
    }
    if (from_host) {
      uint16_t* dp = (uint16_t*)(slot + a.lay.gu_scale_off) + (int64_t)i * 2 * G;
      for (int j = lane; j < 2 * G; j += 32) dp[j] = __ldg(sp + j);
    }
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
#pragma unroll 1
  for (int t = 0; t < tg; t++) {
    const uint8_t* xt = xs + (int64_t)t * xpad;
#pragma unroll
    for (int j = 0; j < CH; j++) {
      opaque(wg[j]);
      opaque(wu[j]);
    }
    float ag = 0.f, au = 0.f;
#pragma unroll
    for (int j = 0; j < CH; j++) {
      const int c = j * 32 + lane;
      if (c < nch) {
        const uint8_t* xc = xt + (int64_t)c * Tr<WD>::xbytes;
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
    if (lane == 0) a.u[(int64_t)pidx[t] * a.I + i] = ag / (1.0f + expf(-ag)) * au;
  }
}

// Stage the activations of pairs plan_tok[off + g0 .. + tg) into xs (one row of xpad bytes each).
__device__ __forceinline__ void stage_x(const BatchArgs& a, int l, int off, int g0, int tg, uint8_t* xs, int xpad,
                                        int* pidx) {
  const int xbytes = a.d * (a.wdtype == WD_FP32 ? 4 : 2);
  const int nq = xbytes / 16;
  if (threadIdx.x < tg) pidx[threadIdx.x] = __ldcg(a.plan_tok + off + g0 + threadIdx.x);
  for (int q = threadIdx.x; q < tg * nq; q += blockDim.x) {
    const int t = q / nq;
    const int c = q - t * nq;
    const int p = __ldcg(a.plan_tok + off + g0 + t);
    const int b = p / a.k;
    const uint4* src = reinterpret_cast<const uint4*>((const uint8_t*)a.hidden + ((int64_t)l * a.B + b) * xbytes);
    *reinterpret_cast<uint4*>(xs + (int64_t)t * xpad + (int64_t)c * 16) = __ldg(src + c);
  }
}

template <int WD, int CH>
__device__ void gateup_item(const BatchArgs& a, int l, int pos, int rblk, bool host_src, uint8_t* smem, int* pidx,
                            int tgmax) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int xpad = (a.d * (WD == WD_FP32 ? 4 : 2) + 15) & ~15;
  const int gid = __ldcg(a.plan_gid + pos);
  const int off = __ldcg(a.plan_off + pos);
  const int cnt = __ldcg(a.plan_cnt + pos);
  uint8_t* slot = a.pool + (int64_t)__ldcg(a.plan_slot + pos) * a.slot_stride;
  const uint8_t* host = a.arena + (int64_t)gid * a.slot_stride;
  const int i0 = rblk * kRowsGU;
  const int i1 = i0 + kRowsGU < a.I ? i0 + kRowsGU : a.I;
  for (int g0 = 0; g0 < cnt; g0 += tgmax) {
    const int tg = cnt - g0 < tgmax ? cnt - g0 : tgmax;
    __syncthreads();  // the previous group's readers are done with xs
    stage_x(a, l, off, g0, tg, smem, xpad, pidx);
    __syncthreads();
    const bool from_host = host_src && g0 == 0;  // later groups reread the rows from the slot
    for (int i = i0 + warp; i < i1; i += kBWarps)
      gateup_rows<WD, CH>(a, from_host ? host : slot, slot, from_host, smem, xpad, pidx, tg, i, lane);
  }
  if (host_src) {
    // this item's share of the expert's W_d region (and int4 scales): a plain copy host -> slot
    const int nrb = (a.I + kRowsGU - 1) / kRowsGU;
    const int64_t nq = (a.lay.total - a.lay.d_off) / 16;
    const int64_t q0 = nq * rblk / nrb, q1 = nq * (rblk + 1) / nrb;
    const uint8_t* src = host + a.lay.d_off;
    uint8_t* dst = slot + a.lay.d_off;
    const int T = blockDim.x;
    int64_t q = q0 + threadIdx.x;
    for (; q + 3 * (int64_t)T < q1; q += 4 * (int64_t)T) {
      const uint4 v0 = ld_stream(src + q * 16);
      const uint4 v1 = ld_stream(src + (q + T) * 16);
      const uint4 v2 = ld_stream(src + (q + 2 * (int64_t)T) * 16);
      const uint4 v3 = ld_stream(src + (q + 3 * (int64_t)T) * 16);
      st_v4(dst + q * 16, v0);
      st_v4(dst + (q + T) * 16, v1);
      st_v4(dst + (q + 2 * (int64_t)T) * 16, v2);
      st_v4(dst + (q + 3 * (int64_t)T) * 16, v3);
    }
    for (; q < q1; q += T) st_v4(dst + q * 16, ld_stream(src + q * 16));
  }
}

// ---- phase D: KR rows of W_d (o, o + 8, ...) applied to the tg staged u vectors
template <int WD, int CHD>
__device__ void down_item(const BatchArgs& a, int pos, int oblk, float* us, int* pidx, int tgmax) {
  constexpr int EPC = Tr<WD>::epc;
  constexpr int KR = 16 / CHD > 4 ? 4 : (16 / CHD < 1 ? 1 : 16 / CHD);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t rb = a.lay.row_bytes_d;
  const int nch = (int)(rb / 16);
  const int G = a.I / 128;
  const int ipad = ipad_of(a.I);
  const int off = __ldcg(a.plan_off + pos);
  const int cnt = __ldcg(a.plan_cnt + pos);
  const uint8_t* slot = a.pool + (int64_t)__ldcg(a.plan_slot + pos) * a.slot_stride;
  const int o0 = oblk * kRowsD;
  const int o1 = o0 + kRowsD < a.d ? o0 + kRowsD : a.d;
  for (int g0 = 0; g0 < cnt; g0 += tgmax) {
    const int tg = cnt - g0 < tgmax ? cnt - g0 : tgmax;
    __syncthreads();
    if (threadIdx.x < tg) pidx[threadIdx.x] = __ldcg(a.plan_tok + off + g0 + threadIdx.x);
    __syncthreads();
    for (int q = threadIdx.x; q < tg * a.I; q += blockDim.x) {
      const int t = q / a.I;
      const int i = q - t * a.I;
      us[t * ipad + upad(i)] = __ldcg(a.u + (int64_t)pidx[t] * a.I + i);
    }
    __syncthreads();
    for (int ob = o0 + warp; ob < o1; ob += kBWarps * KR) {
      uint4 w[KR][CHD];
      float sc[KR][CHD];
#pragma unroll
      for (int rr = 0; rr < KR; rr++) {
        const int o = ob + rr * kBWarps;
        const bool ok = o < o1;
        const int64_t roff = a.lay.d_off + (int64_t)(ok ? o : o0) * rb;
#pragma unroll
        for (int j = 0; j < CHD; j++) {
          const int c = j * 32 + lane;
          w[rr][j] = (ok && c < nch) ? ld_cg(slot + roff + (int64_t)c * 16) : make_uint4(0, 0, 0, 0);
        }
        if (WD == WD_INT4) {
          const uint16_t* sp = (const uint16_t*)(slot + a.lay.d_scale_off) + (int64_t)(ok ? o : o0) * G;
#pragma unroll
          for (int j = 0; j < CHD; j++) {
            const int c = j * 32 + lane;
            sc[rr][j] = (ok && c < nch) ? bf16_bits(__ldcg(sp + (c >> 2))) : 0.f;
          }
        }
      }
#pragma unroll 1
      for (int t = 0; t < tg; t++) {
        const float* ut = us + t * ipad;
#pragma unroll
        for (int rr = 0; rr < KR; rr++)
#pragma unroll
          for (int j = 0; j < CHD; j++) opaque(w[rr][j]);
#pragma unroll
        for (int rr = 0; rr < KR; rr++) {
          float part = 0.f;
#pragma unroll
          for (int j = 0; j < CHD; j++) {
            const int c = j * 32 + lane;
            if (c < nch) {
              if (WD == WD_INT4)
                part = fmaf(sc[rr][j], dot_chunk_u<WD>(w[rr][j], ut + upad(c * EPC), 0.f), part);
              else
                part = dot_chunk_u<WD>(w[rr][j], ut + upad(c * EPC), part);
            }
          }
          part = warp_sum(part);
          const int o = ob + rr * kBWarps;
          if (lane == 0 && o < o1) a.y[(int64_t)pidx[t] * a.d + o] = part;
        }
      }
    }
  }
}

// ---- phase R for all CTAs: items (block of a.router_tb sequences, block of 8 router rows)
__device__ __forceinline__ void phase_router(const BatchArgs& a, int l, uint8_t* xs) {
  // router-guided: phase T folds every sequence's ranks into rank_best (the previous layer-step's
  // phase S has read it)
  if (a.policy == 2 && blockIdx.x == 0)
    for (int e = threadIdx.x; e < a.E; e += blockDim.x) a.rank_best[e] = a.E;
  const int rtb = a.router_tb;
  const int ntb = (a.B + rtb - 1) / rtb;
  const int neb = (a.E + kBWarps - 1) / kBWarps;
  for (int it = blockIdx.x; it < ntb * neb; it += gridDim.x) {
    const int eb = it / ntb, tb = it - eb * ntb;
    if (a.wdtype == WD_FP32)
      router_block<WD_FP32>(a, l, tb, eb, rtb, xs);
    else
      router_block<WD_BF16>(a, l, tb, eb, rtb, xs);
  }
}

// Router-guided policy: every expert's rank in one sequence's routing (the logits that beat its own,
// ties to the lower id, in the top-k's order), folded into the layer-step's best rank over the
// batch. One warp; lane holds experts lane, lane + 32, ... (E <= 256).
__device__ __forceinline__ void fold_ranks(const BatchArgs& a, const float* z, int lane) {
  constexpr int PER = 8;
  uint32_t key[PER];
  int rank[PER];
#pragma unroll
  for (int q = 0; q < PER; q++) {
    const int e = q * 32 + lane;
    key[q] = e < a.E ? ord_key(__ldcg(z + e)) : 0u;
    rank[q] = 0;
  }
#pragma unroll
  for (int qj = 0; qj < PER; qj++) {
    if (qj * 32 >= a.E) break;
    for (int src = 0; src < 32; src++) {
      const int j = qj * 32 + src;
      const uint32_t kj = __shfl_sync(kFull, key[qj], src);
      if (j < a.E) {
#pragma unroll
        for (int q = 0; q < PER; q++) {
          const int e = q * 32 + lane;
          rank[q] += (kj > key[q] || (kj == key[q] && j < e)) ? 1 : 0;
        }
      }
    }
  }
#pragma unroll
  for (int q = 0; q < PER; q++) {
    const int e = q * 32 + lane;
    if (e < a.E) atomicMin(a.rank_best + e, rank[q]);
  }
}

// ---- phase T: one warp per sequence
__device__ __forceinline__ void phase_topk(const BatchArgs& a, int l, int gw, int W, int lane) {
  for (int b = gw; b < a.B; b += W) {
    int my_i;
    float my_g;
    const float* zb = a.z + ((int64_t)l * a.Bmax + b) * a.E;
    warp_topk(zb, a.E, a.k, a.renorm, lane, my_i, my_g);
    if (a.policy == 2) fold_ranks(a, zb, lane);
    if (lane < a.k) {
      if (my_i < 0 || my_i >= a.E) {
        atomicOr(a.err, FERR_BAD_ROUTE);
        my_i = lane;  // keep the step well-defined; the host reports the error
      }
      a.sel_e[b * a.k + lane] = my_i;
      a.sel_g[b * a.k + lane] = my_g;
      a.route_idx[((int64_t)l * a.Bmax + b) * a.k + lane] = my_i;
      a.route_gate[((int64_t)l * a.Bmax + b) * a.k + lane] = my_g;
    }
  }
}

// ---- phase E: out[b][o] = sum_r g_{b,r} y_{b*k+r}[o], ranks in order; four outputs per thread
// (d is a multiple of 4)
__device__ __forceinline__ void phase_combine(const BatchArgs& a, int l) {
  const int d4 = a.d / 4;
  const int64_t nout = (int64_t)a.B * d4;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nout; q += (int64_t)gridDim.x * blockDim.x) {
    const int b = (int)(q / d4);
    const int o = 4 * (int)(q - (int64_t)b * d4);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int r = 0; r < a.k; r++) {
      const int p = b * a.k + r;
      const float g = __ldcg(a.sel_g + p);
      const float4 y = __ldcg(reinterpret_cast<const float4*>(a.y + (int64_t)p * a.d + o));
      acc.x = fmaf(g, y.x, acc.x);
      acc.y = fmaf(g, y.y, acc.y);
      acc.z = fmaf(g, y.z, acc.z);
      acc.w = fmaf(g, y.w, acc.w);
    }
    const int64_t oi = ((int64_t)l * a.B + b) * a.d + o;
    if (a.wdtype == WD_FP32) {
      *reinterpret_cast<float4*>(reinterpret_cast<float*>(a.out) + oi) = acc;
    } else {
      __nv_bfloat162* dst = reinterpret_cast<__nv_bfloat162*>(reinterpret_cast<__nv_bfloat16*>(a.out) + oi);
      dst[0] = __floats2bfloat162_rn(acc.x, acc.y);
      dst[1] = __floats2bfloat162_rn(acc.z, acc.w);
    }
  }
}

// Next work item of a phase for the whole CTA (thread 0 draws it from the phase's counter).
__device__ __forceinline__ int next_item(unsigned* ctr, int* s_item) {
  __syncthreads();  // every thread has read the previous item
  if (threadIdx.x == 0) *s_item = (int)atomicAdd(ctr, 1u);
  __syncthreads();
  return *s_item;
}

template <int WD, int CH>
__global__ void __launch_bounds__(kBThreads, 2) k_fused_batched(const __grid_constant__ BatchArgs a) {
  extern __shared__ uint4 smem4[];
  __shared__ int pidx[kTGMax];
  __shared__ int s_item;
  uint8_t* smem = reinterpret_cast<uint8_t*>(smem4);
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kBWarps + warp;
  const int W = gridDim.x * kBWarps;
  const int64_t step = *(volatile int64_t*)a.step;
  const int tgmax = a.tg_max;
  const int chd_need = (int)((a.lay.row_bytes_d / 16 + 31) / 32);
  const int nrb = (a.I + kRowsGU - 1) / kRowsGU;
  const int nob = (a.d + kRowsD - 1) / kRowsD;
  unsigned nbar = 0;
  if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[a.L * kBatchedPhases] = gtimer();
  auto mark = [&](int l, int ph) {
    if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[l * kBatchedPhases + ph] = gtimer();
  };

  for (int l = 0; l < a.L; l++) {
    const int clock = (int)(step * a.L + l + 1);  // 0 is older than every step (preloaded experts)
    phase_router(a, l, smem);
    if (!grid_sync(a, nbar)) return;
    mark(l, 0);
    phase_topk(a, l, gw, W, lane);
    if (!grid_sync(a, nbar)) return;
    mark(l, 1);
    // ---- S
    if (blockIdx.x == 0) batched_select(a, l, clock, step, reinterpret_cast<unsigned long long*>(smem));
    if (!grid_sync(a, nbar)) return;
    mark(l, 2);
    // ---- C
    {
      const int n = __ldcg(a.plan_n);
      const int nm = __ldcg(a.plan_n + 1);
      if (nm > 0) {
        // warm the host-link address translations of every missed expert (one L2 prefetch per page)
        const int64_t pages = (a.lay.total + (1 << a.touch_shift) - 1) >> a.touch_shift;
        const int64_t gt0 = (int64_t)blockIdx.x * kBThreads + threadIdx.x;
        const int64_t GT = (int64_t)gridDim.x * kBThreads;
        for (int64_t q = gt0; q < (int64_t)nm * pages; q += GT) {
          const int m = (int)(q / pages);
          const uint8_t* pa =
              a.arena + (int64_t)__ldcg(a.plan_gid + m) * a.slot_stride + ((q - (int64_t)m * pages) << a.touch_shift);
          asm volatile("prefetch.global.L2 [%0];" ::"l"(pa));
        }
      }
      // items: plan position (misses first) x row block
      for (int it = next_item(a.work, &s_item); it < n * nrb; it = next_item(a.work, &s_item)) {
        const int pos = it / nrb;
        gateup_item<WD, CH>(a, l, pos, it - pos * nrb, pos < nm, smem, pidx, tgmax);
      }
    }
    if (!grid_sync(a, nbar)) return;
    mark(l, 3);
    // ---- D
    {
      const int n = __ldcg(a.plan_n);
      float* us = reinterpret_cast<float*>(smem);
      for (int it = next_item(a.work + 1, &s_item); it < n * nob; it = next_item(a.work + 1, &s_item)) {
        const int pos = it / nob, ob = it % nob;
        switch (chd_need) {
          case 1: down_item<WD, 1>(a, pos, ob, us, pidx, tgmax); break;
          case 2: down_item<WD, 2>(a, pos, ob, us, pidx, tgmax); break;
          case 3: down_item<WD, 3>(a, pos, ob, us, pidx, tgmax); break;
          case 4: down_item<WD, 4>(a, pos, ob, us, pidx, tgmax); break;
          case 5:
          case 6: down_item<WD, 6>(a, pos, ob, us, pidx, tgmax); break;
          default: down_item<WD, 8>(a, pos, ob, us, pidx, tgmax); break;
        }
      }
    }
    if (!grid_sync(a, nbar)) return;
    mark(l, 4);
    phase_combine(a, l);
    if (!grid_sync(a, nbar)) return;
    mark(l, 5);
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) *a.step = step + 1;
}

// =============================================================================================
// Tensor-core variant (bf16 weights). Phases C and D become grouped GEMMs on tcgen05: a work item
// is (needed expert, 128-row tile of its weight matrix); the A operand (weights, 128 rows x 64 K
// per stage) and the B operand (the expert's pairs, N = pair count rounded up to 16 rows x 64 K)
// stream from global memory into a ring of shared-memory stages by TMA; one thread issues the
// MMAs (M = 128, N, K = 16) into a TMEM accumulator; four epilogue warps read the accumulator
// back (TMEM lane = weight row, column = pair). Per CTA: warp 0 lane 0 produces, warp 1 lane 0
// issues MMAs, warps 4-7 run the epilogue, two accumulators alternate so the epilogue of one
// item overlaps the MMAs of the next. Missed experts are copied host -> slot in the phase before
// (G), so every expert's arithmetic is the same whether it hit or missed.

constexpr int kTcStages = 6;
constexpr int kTcABytes = 128 * 64 * 2;             // one A stage: 128 rows x 64 bf16
constexpr int kTcStageBytes = kTcABytes + 64 * 128; // + up to 64 B-operand rows of 128 B
constexpr int kTcAccCols = 64;                      // fp32 columns per accumulator (N <= 64)
constexpr int kTcTmemCols = 2 * kTcAccCols;
constexpr int kTcCopyChunk = 256 * 1024;            // bytes per miss-copy work item
constexpr unsigned long long kPipeTimeoutNs = 2000000000ull;

struct TcShared {
  uint64_t full[kTcStages];   // stage loaded (TMA transaction bytes)
  uint64_t empty[kTcStages];  // stage consumed (tcgen05.commit)
  uint64_t accfull[2];        // accumulator complete (tcgen05.commit)
  uint64_t accempty[2];       // accumulator read back (4 epilogue warps)
  uint32_t tmem;
};

// Position in the stage ring and the accumulator pair; the producer, the MMA thread and the
// epilogue threads each keep a copy and advance it over the same item sequence.
struct TcRing {
  uint32_t stage = 0, sphase = 0, acc = 0, aphase = 0;
  __device__ void next_stage() {
    if (++stage == kTcStages) {
      stage = 0;
      sphase ^= 1u;
    }
  }
  __device__ void next_acc() {
    if (++acc == 2) {
      acc = 0;
      aphase ^= 1u;
    }
  }
};

struct TcGemm {
  const CUtensorMap* map_a;  // weights in the slot pool (3D: K, row, slot)
  const CUtensorMap* map_b;  // pairs in plan order (2D: K, row)
  int mtiles;                // 128-row tiles per expert
  int nkb;                   // 64-wide K blocks
};

__device__ __forceinline__ bool tc_wait(const BatchArgs& a, uint64_t* bar, uint32_t parity) {
  if (tc::mbar_wait(bar, parity, kPipeTimeoutNs, a.err, FERR_FATAL)) return true;
  atomicOr(a.err, FERR_PIPE_TIMEOUT);
  return false;
}

__device__ void tc_produce(const BatchArgs& a, TcShared& st, const TcGemm& g, int nitems, uint8_t* stages,
                           TcRing& r) {
  tc::fence_proxy_async_global();  // the B rows (and missed experts) were written by ordinary stores
  for (int it = blockIdx.x; it < nitems; it += gridDim.x) {
    const int pos = it / g.mtiles, mt = it - pos * g.mtiles;
    const int slot = __ldcg(a.plan_slot + pos), off = __ldcg(a.plan_off + pos), cnt = __ldcg(a.plan_cnt + pos);
    const int nb16 = (cnt + 15) >> 4;
    for (int kb = 0; kb < g.nkb; kb++) {
      if (!tc_wait(a, &st.empty[r.stage], r.sphase ^ 1u)) return;
      uint8_t* sa = stages + r.stage * kTcStageBytes;
      tc::mbar_expect_tx(&st.full[r.stage], (uint32_t)(kTcABytes + nb16 * 2048));
      tc::tma_load_3d(sa, g.map_a, &st.full[r.stage], kb * 64, mt * 128, slot);
      for (int j = 0; j < nb16; j++)
        tc::tma_load_2d(sa + kTcABytes + j * 2048, g.map_b, &st.full[r.stage], kb * 64, off + 16 * j);
      r.next_stage();
    }
  }
}

__device__ void tc_mma(const BatchArgs& a, TcShared& st, const TcGemm& g, int nitems, uint8_t* stages, TcRing& r) {
  for (int it = blockIdx.x; it < nitems; it += gridDim.x) {
    const int pos = it / g.mtiles;
    const int cnt = __ldcg(a.plan_cnt + pos);
    const uint32_t idesc = tc::idesc_bf16(128, ((cnt + 15) >> 4) * 16);
    if (!tc_wait(a, &st.accempty[r.acc], r.aphase ^ 1u)) return;
    tc::fence_after_sync();
    const uint32_t d = st.tmem + r.acc * kTcAccCols;
    for (int kb = 0; kb < g.nkb; kb++) {
      if (!tc_wait(a, &st.full[r.stage], r.sphase)) return;
      tc::fence_after_sync();
      const uint32_t sa = tc::smem_u32(stages + r.stage * kTcStageBytes);
      const uint64_t da = tc::desc_sw128(sa), db = tc::desc_sw128(sa + kTcABytes);
#pragma unroll
      for (int j = 0; j < 4; j++)  // K = 16 per MMA: the next 32 B of every 128-B row
        tc::mma_bf16(d, da + (uint64_t)(2 * j), db + (uint64_t)(2 * j), idesc, (kb | j) != 0);
      tc::mma_commit(&st.empty[r.stage]);
      r.next_stage();
    }
    tc::mma_commit(&st.accfull[r.acc]);
    r.next_acc();
  }
}

// Epilogue warps 4-7: warp q = warp % 4 reads TMEM lanes [32q, 32q + 32), i.e. weight rows
// mt * 128 + 32q + lane, 16 pair columns at a time; f consumes them.
template <typename F>
__device__ void tc_epilogue(const BatchArgs& a, TcShared& st, const TcGemm& g, int nitems, TcRing& r, F&& f) {
  const int q = (threadIdx.x >> 5) & 3, lane = threadIdx.x & 31;
  for (int it = blockIdx.x; it < nitems; it += gridDim.x) {
    const int pos = it / g.mtiles, mt = it - pos * g.mtiles;
    const int off = __ldcg(a.plan_off + pos), cnt = __ldcg(a.plan_cnt + pos);
    if (!tc_wait(a, &st.accfull[r.acc], r.aphase)) return;
    tc::fence_after_sync();
    const uint32_t t0 = st.tmem + r.acc * kTcAccCols + ((uint32_t)(q * 32) << 16);
    const int row = mt * 128 + q * 32 + lane;
    for (int c0 = 0; c0 < cnt; c0 += 16) {
      float v[16];
      tc::tmem_ld16(t0 + (uint32_t)c0, v);
      f(off, cnt, row, c0, v, lane);
    }
    tc::fence_before_sync();
    __syncwarp();
    if (lane == 0) tc::mbar_arrive(&st.accempty[r.acc]);
    r.next_acc();
  }
}

// ---- phase G: the pairs' activations into plan order (xg), and every missed expert's image
// host -> slot (chunks handed out dynamically, after a translation warm-up as in phase C of the
// CUDA-core variant).
__device__ void tc_gather_copy(const BatchArgs& a, int l, int gw, int W, int lane, int* s_item) {
  const int nm = __ldcg(a.plan_n + 1);
  const int P = a.B * a.k;
  if (nm > 0 && a.touch_shift > 0) {
    const int64_t pages = (a.lay.total + (1 << a.touch_shift) - 1) >> a.touch_shift;
    const int64_t gt0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t GT = (int64_t)gridDim.x * blockDim.x;
    for (int64_t q = gt0; q < (int64_t)nm * pages; q += GT) {
      const int m = (int)(q / pages);
      const uint8_t* pa =
          a.arena + (int64_t)__ldcg(a.plan_gid + m) * a.slot_stride + ((q - (int64_t)m * pages) << a.touch_shift);
      asm volatile("prefetch.global.L2 [%0];" ::"l"(pa));
    }
  }
  const int nq = a.d * 2 / 16;
  for (int j = gw; j < P; j += W) {
    const int b = __ldcg(a.plan_tok + j) / a.k;
    const uint4* src = reinterpret_cast<const uint4*>((const uint8_t*)a.hidden + ((int64_t)l * a.B + b) * a.d * 2);
    uint8_t* dst = reinterpret_cast<uint8_t*>(a.xg) + (int64_t)j * a.d * 2;
    for (int c = lane; c < nq; c += 32) st_v4(dst + c * 16, __ldg(src + c));
  }
  const int cpe = (int)((a.lay.total + kTcCopyChunk - 1) / kTcCopyChunk);
  for (int it = next_item(a.work, s_item); it < nm * cpe; it = next_item(a.work, s_item)) {
    const int m = it / cpe, c = it - m * cpe;
    const int64_t b0 = (int64_t)c * kTcCopyChunk;
    const int64_t b1 = b0 + kTcCopyChunk < a.lay.total ? b0 + kTcCopyChunk : a.lay.total;
    const uint8_t* src = a.arena + (int64_t)__ldcg(a.plan_gid + m) * a.slot_stride;
    uint8_t* dst = a.pool + (int64_t)__ldcg(a.plan_slot + m) * a.slot_stride;
    const int T = blockDim.x;
    int64_t q = b0 / 16 + threadIdx.x;
    const int64_t q1 = b1 / 16;
    for (; q + 3 * (int64_t)T < q1; q += 4 * (int64_t)T) {
      const uint4 v0 = ld_stream(src + q * 16);
      const uint4 v1 = ld_stream(src + (q + T) * 16);
      const uint4 v2 = ld_stream(src + (q + 2 * (int64_t)T) * 16);
      const uint4 v3 = ld_stream(src + (q + 3 * (int64_t)T) * 16);
      st_v4(dst + q * 16, v0);
      st_v4(dst + (q + T) * 16, v1);
      st_v4(dst + (q + 2 * (int64_t)T) * 16, v2);
      st_v4(dst + (q + 3 * (int64_t)T) * 16, v3);
    }
    for (; q < q1; q += T) st_v4(dst + q * 16, ld_stream(src + q * 16));
  }
}

__global__ void __launch_bounds__(kBThreads, 1) k_fused_batched_tc(const __grid_constant__ BatchArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  __shared__ TcShared st;
  __shared__ int s_item;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kBWarps + warp;
  const int W = gridDim.x * kBWarps;
  const int64_t step = *(volatile int64_t*)a.step;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kTcStages; i++) {
      tc::mbar_init(&st.full[i], 1);
      tc::mbar_init(&st.empty[i], 1);
    }
    for (int i = 0; i < 2; i++) {
      tc::mbar_init(&st.accfull[i], 1);
      tc::mbar_init(&st.accempty[i], 4);
    }
    tc::fence_mbar_init();
    tc::prefetch_tmap(&a.map_gu);
    tc::prefetch_tmap(&a.map_d);
    tc::prefetch_tmap(&a.map_x);
    tc::prefetch_tmap(&a.map_u);
  }
  if (warp == 2) {
    tc::tmem_alloc(&st.tmem, kTcTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[a.L * kBatchedTcPhases] = gtimer();
  auto mark = [&](int l, int ph) {
    if (a.phase_ts && blockIdx.x == 0 && threadIdx.x == 0) a.phase_ts[l * kBatchedTcPhases + ph] = gtimer();
  };
  const TcGemm gu{&a.map_gu, &a.map_x, 2 * a.I / 128, a.d / 64};
  const TcGemm dn{&a.map_d, &a.map_u, a.d / 128, a.I / 64};
  TcRing ring;
  unsigned nbar = 0;

  auto layers = [&]() -> bool {
    for (int l = 0; l < a.L; l++) {
      const int clock = (int)(step * a.L + l + 1);
      phase_router(a, l, smem);
      if (!grid_sync(a, nbar)) return false;
      mark(l, 0);
      phase_topk(a, l, gw, W, lane);
      if (!grid_sync(a, nbar)) return false;
      mark(l, 1);
      if (blockIdx.x == 0) batched_select(a, l, clock, step, reinterpret_cast<unsigned long long*>(smem));
      if (!grid_sync(a, nbar)) return false;
      mark(l, 2);
      tc_gather_copy(a, l, gw, W, lane, &s_item);
      tc::fence_proxy_async_global();
      if (!grid_sync(a, nbar)) return false;
      mark(l, 3);
      // ---- C: [gate; up] rows x pairs -> u = silu(gate) * up, bf16, plan order
      {
        const int items = __ldcg(a.plan_n) * gu.mtiles;
        if (warp == 0) {
          if (lane == 0) tc_produce(a, st, gu, items, smem, ring);
        } else if (warp == 1) {
          if (lane == 0) tc_mma(a, st, gu, items, smem, ring);
        } else if (warp >= 4) {
          tc_epilogue(a, st, gu, items, ring, [&](int off, int cnt, int row, int c0, float(&v)[16], int ln) {
            // rows alternate gate, up of one intermediate index: lanes 2j and 2j + 1 hold a pair
            const int i = row >> 1;
#pragma unroll
            for (int t = 0; t < 16; t++) {
              const float other = __shfl_xor_sync(kFull, v[t], 1);
              if (!(ln & 1) && c0 + t < cnt) {
                const float g = v[t];
                a.ug[(int64_t)(off + c0 + t) * a.I + i] = __float2bfloat16_rn(g / (1.0f + expf(-g)) * other);
              }
            }
          });
        }
      }
      tc::fence_proxy_async_global();
      if (!grid_sync(a, nbar)) return false;
      mark(l, 4);
      // ---- D: W_d rows x pairs -> y[pair][row]
      {
        const int items = __ldcg(a.plan_n) * dn.mtiles;
        if (warp == 0) {
          if (lane == 0) tc_produce(a, st, dn, items, smem, ring);
        } else if (warp == 1) {
          if (lane == 0) tc_mma(a, st, dn, items, smem, ring);
        } else if (warp >= 4) {
          tc_epilogue(a, st, dn, items, ring, [&](int off, int cnt, int row, int c0, float(&v)[16], int) {
#pragma unroll
            for (int t = 0; t < 16; t++)
              if (c0 + t < cnt) a.y[(int64_t)__ldcg(a.plan_tok + off + c0 + t) * a.d + row] = v[t];
          });
        }
      }
      if (!grid_sync(a, nbar)) return false;
      mark(l, 5);
      phase_combine(a, l);
      if (!grid_sync(a, nbar)) return false;
      mark(l, 6);
    }
    return true;
  };
  const bool ok = layers();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (warp == 2) tc::tmem_dealloc(st.tmem, kTcTmemCols);
  if (ok && blockIdx.x == 0 && threadIdx.x == 0) *a.step = step + 1;
}

size_t batched_tc_smem(int64_t cap, int64_t n_gid) {
  return std::max((size_t)kTcStages * kTcStageBytes, (size_t)sort_n_of(cap, n_gid) * sizeof(unsigned long long)) +
         1024;
}

int pick_ch_b(int64_t rb) {
  const int need = (int)((rb / 16 + 31) / 32);
  if (need <= 1) return 1;
  if (need <= 2) return 2;
  if (need <= 4) return 4;
  if (need <= 8) return 8;
  if (need <= 16) return 16;
  return -1;
}

template <int WD, int CH>
int grid_of_b(size_t smem) {
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(k_fused_batched<WD, CH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
          cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_fused_batched<WD, CH>, kBThreads, smem) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms * (occ < 2 ? occ : 2);
}

template <int WD, int CH>
cudaError_t run_fused_b(const BatchArgs& a, int grid, cudaStream_t s) {
  const size_t smem = batched_smem(a.wdtype, a.d, a.I, a.cap, a.n_gid);
  void* params[] = {(void*)&a};
  return cudaLaunchCooperativeKernel((const void*)k_fused_batched<WD, CH>, dim3(grid), dim3(kBThreads), params, smem,
                                     s);
}

}  // namespace

#define MOE_B_DISPATCH(FN, WDV, CHV, ...)               \
  do {                                                  \
    switch (WDV) {                                      \
      case WD_FP32:                                     \
        switch (CHV) {                                  \
          case 1: return FN<WD_FP32, 1>(__VA_ARGS__);   \
          case 2: return FN<WD_FP32, 2>(__VA_ARGS__);   \
          case 4: return FN<WD_FP32, 4>(__VA_ARGS__);   \
          case 8: return FN<WD_FP32, 8>(__VA_ARGS__);   \
        }                                               \
        break;                                          \
      case WD_BF16:                                     \
        switch (CHV) {                                  \
          case 1: return FN<WD_BF16, 1>(__VA_ARGS__);   \
          case 2: return FN<WD_BF16, 2>(__VA_ARGS__);   \
          case 4: return FN<WD_BF16, 4>(__VA_ARGS__);   \
          case 8: return FN<WD_BF16, 8>(__VA_ARGS__);   \
          case 16: return FN<WD_BF16, 16>(__VA_ARGS__); \
        }                                               \
        break;                                          \
      case WD_INT4:                                     \
        switch (CHV) {                                  \
          case 1: return FN<WD_INT4, 1>(__VA_ARGS__);   \
          case 2: return FN<WD_INT4, 2>(__VA_ARGS__);   \
          case 4: return FN<WD_INT4, 4>(__VA_ARGS__);   \
          case 8: return FN<WD_INT4, 8>(__VA_ARGS__);   \
        }                                               \
        break;                                          \
    }                                                   \
  } while (0)

int batched_tg(int wdtype, int d, int I) { return tg_of(wdtype, d, I); }

int batched_router_tb(int wdtype, int d, int I, bool tensor_cores) {
  const int xpad = (d * (wdtype == WD_FP32 ? 4 : 2) + 15) & ~15;
  // the dynamic shared memory without the sort keys (which may be absent)
  const size_t smem = tensor_cores ? (size_t)kTcStages * kTcStageBytes
                                   : (size_t)tg_of(wdtype, d, I) * std::max(xpad, ipad_of(I) * 4);
  return (int)std::max<size_t>(1, std::min<size_t>(8, smem / xpad));
}

int fused_batched_grid(int wdtype, int d, int I, int64_t cap, int64_t n_gid) {
  if (sort_n_of(cap, n_gid) > kBatchedEvictCap) return 0;
  const BlobLayout lay = make_layout(wdtype, d, I);
  const int ch = pick_ch_b(lay.row_bytes_gu);
  const size_t smem = batched_smem(wdtype, d, I, cap, n_gid);
  if (smem > 200 * 1024) return 0;
  MOE_B_DISPATCH(grid_of_b, wdtype, ch, smem);
  return 0;
}

cudaError_t launch_fused_batched(const BatchArgs& a, int grid, cudaStream_t s) {
  const int ch = pick_ch_b(a.lay.row_bytes_gu);
  MOE_B_DISPATCH(run_fused_b, a.wdtype, ch, a, grid, s);
  return cudaErrorInvalidValue;
}

bool batched_tc_supported(int wdtype, int d, int I) {
  return wdtype == WD_BF16 && d % 128 == 0 && I % 64 == 0 && d <= 16384 && I <= 16384;
}

int fused_batched_tc_grid(int d, int I, int64_t cap, int64_t n_gid) {
  if (!batched_tc_supported(WD_BF16, d, I) || sort_n_of(cap, n_gid) > kBatchedEvictCap) return 0;
  const size_t smem = batched_tc_smem(cap, n_gid);
  if (cudaFuncSetAttribute(k_fused_batched_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_fused_batched_tc, kBThreads, smem) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return occ >= 1 ? sms : 0;  // one CTA per SM: its TMEM allocation never waits on another CTA's
}

cudaError_t launch_fused_batched_tc(const BatchArgs& a, int grid, cudaStream_t s) {
  const size_t smem = batched_tc_smem(a.cap, a.n_gid);
  void* params[] = {(void*)&a};
  return cudaLaunchCooperativeKernel((const void*)k_fused_batched_tc, dim3(grid), dim3(kBThreads), params, smem, s);
}

}  // namespace moe
