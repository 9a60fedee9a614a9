/*
 * fp64 CPU oracle of the capped-residency MoE decode step.
 *
 * TEST INFRASTRUCTURE ONLY: nothing on the product path may call this code. It
 * is used by the tests, by __graft_entry__.smoke() to check the CUDA path, and
 * by bench.py's CPU-baseline leg. It shares no code with the CUDA library.
 *
 * The method (paper, Section "Rotary GPU Concept" and Fig. 1): full expert
 * weights stay in a host tier; a fixed group of accelerator slots holds a
 * subset of sub-modules (experts); a lookup table maps sub-module id -> slot;
 * the routing result (hidden state h, routing vector r) drives residency;
 * missing sub-modules are loaded selectively, residents are evicted. The
 * paper does not disclose its replacement policy, so the residency step here
 * is a deterministic LRU with lower-id ties (see orc_lru_step).
 *
 * Contents, in file order:
 *   widening of stored weights; matvec, softmax, top-k, the router; the SwiGLU
 *     expert FFN and the combine (one MoE layer);
 *   residency steps: LRU (orc_lru_step), our reading of the rotary slot group
 *     (orc_rotary_step, Fig. 1/2), prefetch admission after an LRU step
 *     (orc_lru_admit) and router-guided replacement (orc_guided_step), the
 *     last two readings of the paper's residency decisions that use
 *     information produced during execution (Sec. 3);
 *   the decoder block around the MoE layer: RMSNorm, rotary positions and
 *     grouped-query attention over a KV cache (orc_rmsnorm, orc_rope,
 *     orc_attend), chained by oracle/decoder.py.
 *
 * Everything is plain fp64 arithmetic on exactly widened inputs, one rounded
 * operation at a time (built with -ffp-contract=off, no fast-math), sums in
 * ascending index order. Rows of a matrix-vector product may be spread over
 * OpenMP threads; each dot product is still one sequential sum, so the result
 * does not depend on the thread count.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* Storage codes of weights and activations. */
enum { ORC_FP32 = 0, ORC_BF16 = 1, ORC_INT4_G128 = 2 };

static double bf16_bits_to_double(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

/*
 * Exact widening of a stored [rows x cols] matrix to fp64.
 *   fp32, bf16: the stored value.
 *   int4 g128:  q * s, q the signed nibble (element 2j = low nibble of byte j
 *               of the row, two's complement), s the bf16 scale of the group of
 *               128 consecutive elements of the row that holds the element.
 * Returns 0, or -1 for an unknown code / int4 cols not a multiple of 128.
 */
int orc_widen(int dtype, const void* src, const uint16_t* scales, int64_t rows, int64_t cols, double* dst) {
  if (dtype == ORC_FP32) {
    const float* s = (const float*)src;
    for (int64_t i = 0; i < rows * cols; i++) dst[i] = (double)s[i];
    return 0;
  }
  if (dtype == ORC_BF16) {
    const uint16_t* s = (const uint16_t*)src;
    for (int64_t i = 0; i < rows * cols; i++) dst[i] = bf16_bits_to_double(s[i]);
    return 0;
  }
  if (dtype == ORC_INT4_G128) {
    if (cols % 128 != 0) return -1;
    const uint8_t* q = (const uint8_t*)src;
    int64_t groups = cols / 128;
    for (int64_t r = 0; r < rows; r++) {
      for (int64_t c = 0; c < cols; c++) {
        uint8_t byte = q[(r * cols + c) / 2];
        int nib = (c % 2 == 0) ? (byte & 0xF) : (byte >> 4);
        int qv = nib >= 8 ? nib - 16 : nib;
        double s = bf16_bits_to_double(scales[r * groups + c / 128]);
        dst[r * cols + c] = (double)qv * s;
      }
    }
    return 0;
  }
  return -1;
}

/* y = W x for W [rows x cols] row-major: y_i = sum_{j=0..cols-1} W_ij x_j, j ascending. */
void orc_matvec(const double* W, const double* x, int64_t rows, int64_t cols, double* y) {
#pragma omp parallel for schedule(static) if (rows * cols > 65536)
  for (int64_t i = 0; i < rows; i++) {
    const double* w = W + i * cols;
    double acc = 0.0;
    for (int64_t j = 0; j < cols; j++) acc += w[j] * x[j];
    y[i] = acc;
  }
}

/* Softmax over n logits with the maximum subtracted: p_e = exp(z_e - m) / sum_j exp(z_j - m). */
void orc_softmax(const double* z, int64_t n, double* p) {
  double m = z[0];
  for (int64_t e = 1; e < n; e++)
    if (z[e] > m) m = z[e];
  double s = 0.0;
  for (int64_t e = 0; e < n; e++) {
    p[e] = exp(z[e] - m);
    s += p[e];
  }
  for (int64_t e = 0; e < n; e++) p[e] = p[e] / s;
}

/*
 * Top-k by logit: the k largest z, ties broken toward the lower expert id, in
 * output order descending z (equal z: lower id first). Plain repeated
 * selection. `taken` is scratch of n bytes.
 */
void orc_topk(const double* z, int64_t n, int32_t k, int32_t* idx, uint8_t* taken) {
  memset(taken, 0, (size_t)n);
  for (int32_t r = 0; r < k; r++) {
    int64_t best = -1;
    for (int64_t e = 0; e < n; e++) {
      if (taken[e]) continue;
      if (best < 0 || z[e] > z[best]) best = e;
    }
    taken[best] = 1;
    idx[r] = (int32_t)best;
  }
}

/*
 * Routing result for one hidden vector (the paper's "routing result" driving
 * residency, Fig. 1): logits z = W_r h, probabilities p = softmax(z) over all
 * E experts, top-k ids by z, gates g_r = p_{e_r} / sum_{j<k} p_{e_j} (renorm=1)
 * or g_r = p_{e_r} (renorm=0).
 * If forced_idx is non-NULL its k ids are taken as the selection (used to
 * re-evaluate a step with another implementation's ids after a near-tie flip).
 * z_out, p_out: optional [E] outputs. scratch: 2E doubles + E bytes.
 */
void orc_router(const double* Wr, const double* h, int32_t E, int32_t d, int32_t k, int32_t renorm,
                const int32_t* forced_idx, int32_t* idx, double* gate, double* z_out, double* p_out,
                double* scratch) {
  double* z = scratch;
  double* p = scratch + E;
  uint8_t* taken = (uint8_t*)(scratch + 2 * E);
  orc_matvec(Wr, h, E, d, z);
  orc_softmax(z, E, p);
  if (forced_idx) {
    for (int32_t r = 0; r < k; r++) idx[r] = forced_idx[r];
  } else {
    orc_topk(z, E, k, idx, taken);
  }
  double s = 0.0;
  for (int32_t r = 0; r < k; r++) s += p[idx[r]];
  for (int32_t r = 0; r < k; r++) gate[r] = renorm ? p[idx[r]] / s : p[idx[r]];
  if (z_out) memcpy(z_out, z, sizeof(double) * (size_t)E);
  if (p_out) memcpy(p_out, p, sizeof(double) * (size_t)E);
}

/*
 * SwiGLU expert FFN on one input x [d]:
 *   a = W_g x, b = W_u x (W_g, W_u [I x d]),
 *   u_i = a_i * sigma(a_i) * b_i with sigma(a) = 1 / (1 + exp(-a)),
 *   y = W_d u (W_d [d x I]).
 * scratch: 3I doubles (a, b, u); u_out optional [I].
 */
void orc_expert_ffn(const double* Wg, const double* Wu, const double* Wd, const double* x, int32_t d, int32_t I,
                    double* y, double* u_out, double* scratch) {
  double* a = scratch;
  double* b = scratch + I;
  double* u = scratch + 2 * I;
  orc_matvec(Wg, x, I, d, a);
  orc_matvec(Wu, x, I, d, b);
  for (int32_t i = 0; i < I; i++) {
    double sig = 1.0 / (1.0 + exp(-a[i]));
    u[i] = a[i] * sig * b[i];
  }
  orc_matvec(Wd, u, d, I, y);
  if (u_out) memcpy(u_out, u, sizeof(double) * (size_t)I);
}

/* Gate-weighted combine in fixed rank order: out = sum_{r=0..k-1} g_r y_r, y [k x d]. */
void orc_combine(const double* y, const double* gate, int32_t k, int32_t d, double* out) {
  for (int32_t i = 0; i < d; i++) {
    double acc = 0.0;
    for (int32_t r = 0; r < k; r++) acc += gate[r] * y[(int64_t)r * d + i];
    out[i] = acc;
  }
}

/* One residency record: a requested expert's outcome in one layer-step. */
typedef struct {
  int32_t step;    /* decode step (token index) */
  int32_t layer;
  int32_t expert;  /* expert id within the layer */
  int32_t kind;    /* 0 hit, 1 miss, 2 prefetch admission (orc_lru_admit) */
  int32_t slot;    /* slot that holds the expert after the step */
  int32_t evicted; /* global id of the evicted expert, -1 if a free slot was used or on a hit */
} orc_rec;

static int in_sorted(const int32_t* a, int32_t n, int32_t v) {
  for (int32_t i = 0; i < n; i++)
    if (a[i] == v) return 1;
  return 0;
}

/*
 * One layer-step of the residency state machine (the slot group + lookup
 * table of Fig. 1, with LRU standing in for the undisclosed rotary policy).
 *
 * State: slot_of[gid] (-1 absent), gid_of[slot] (-1 free), last_use[gid].
 * needed: the distinct global expert ids requested in this layer-step, in
 * ascending order (gid = layer * E + expert). clock: this layer-step's index.
 *
 * For each needed gid in ascending order: if resident, a hit. Otherwise a
 * miss: take the lowest-index free slot if there is one; else evict the
 * resident gid v not in `needed` with the smallest (last_use[v], v), and take
 * v's slot. Every needed gid is pinned for the step (never a victim). After
 * all misses, last_use[x] = clock for every needed x. One record per needed
 * gid, in ascending gid order.
 *
 * Returns the number of records, or -1 if no victim exists (cap < |needed|).
 */
int32_t orc_lru_step(int64_t cap, int32_t* slot_of, int32_t* gid_of, int64_t* last_use, int64_t clock,
                     const int32_t* needed, int32_t n, int32_t n_experts, int32_t step, orc_rec* out) {
  for (int32_t i = 0; i < n; i++) {
    int32_t g = needed[i];
    orc_rec rec;
    rec.step = step;
    rec.layer = g / n_experts;
    rec.expert = g % n_experts;
    if (slot_of[g] >= 0) {
      rec.kind = 0;
      rec.slot = slot_of[g];
      rec.evicted = -1;
    } else {
      int64_t slot = -1;
      for (int64_t s = 0; s < cap; s++) {
        if (gid_of[s] < 0) {
          slot = s;
          break;
        }
      }
      int32_t victim = -1;
      if (slot < 0) {
        for (int64_t s = 0; s < cap; s++) {
          int32_t v = gid_of[s];
          if (v < 0 || in_sorted(needed, n, v)) continue;
          if (victim < 0 || last_use[v] < last_use[victim] || (last_use[v] == last_use[victim] && v < victim)) {
            victim = v;
            slot = s;
          }
        }
        if (victim < 0) return -1;
        slot_of[victim] = -1;
      }
      gid_of[slot] = g;
      slot_of[g] = (int32_t)slot;
      rec.kind = 1;
      rec.slot = (int32_t)slot;
      rec.evicted = victim;
    }
    out[i] = rec;
  }
  for (int32_t i = 0; i < n; i++) last_use[needed[i]] = clock;
  return n;
}

/*
 * One layer-step of the rotary slot group: one reading of the paper's rotary residency
 * (Fig. 1 "Rotary Slot Group", Fig. 2 "cyclical forward and reverse rotation"; the paper gives no
 * algorithm). The cap slots form a ring with a hand; each slot remembers its previous occupant.
 *
 * State: slot_of[gid], gid_of[slot] (-1 empty), prior[slot] (the gid last evicted from the slot,
 * -1 none), *hand (a slot index). needed: distinct gids of the layer-step, ascending.
 *
 * For each needed gid g in ascending order: if resident, a hit (nothing moves). Otherwise a miss:
 *   reverse rotation: if some slot s has prior[s] == g and s holds no gid of `needed`, g returns
 *     to s;
 *   forward rotation: otherwise g takes the first slot s at or after *hand (cyclically) that holds
 *     no gid of `needed`, and *hand moves to s + 1 (mod cap).
 * The occupant v of s (if any) is evicted: slot_of[v] = -1. Then prior[s] = v (possibly -1), every
 * other prior entry equal to g is cleared, and g is placed in s. One record per needed gid.
 *
 * Returns the number of records, or -1 if no slot is available (cap < |needed|).
 */
int32_t orc_rotary_step(int64_t cap, int32_t* slot_of, int32_t* gid_of, int32_t* prior, int64_t* hand,
                        const int32_t* needed, int32_t n, int32_t n_experts, int32_t step, orc_rec* out) {
  for (int32_t i = 0; i < n; i++) {
    int32_t g = needed[i];
    orc_rec rec;
    rec.step = step;
    rec.layer = g / n_experts;
    rec.expert = g % n_experts;
    if (slot_of[g] >= 0) {
      rec.kind = 0;
      rec.slot = slot_of[g];
      rec.evicted = -1;
      out[i] = rec;
      continue;
    }
    int64_t slot = -1;
    for (int64_t s = 0; s < cap; s++) {
      if (prior[s] == g && (gid_of[s] < 0 || !in_sorted(needed, n, gid_of[s]))) {
        slot = s;
        break;
      }
    }
    if (slot < 0) {
      for (int64_t j = 0; j < cap; j++) {
        int64_t s = (*hand + j) % cap;
        if (gid_of[s] < 0 || !in_sorted(needed, n, gid_of[s])) {
          slot = s;
          break;
        }
      }
      if (slot < 0) return -1;
      *hand = (slot + 1) % cap;
    }
    int32_t v = gid_of[slot];
    if (v >= 0) slot_of[v] = -1;
    for (int64_t s = 0; s < cap; s++)
      if (prior[s] == g) prior[s] = -1;
    prior[slot] = v;
    gid_of[slot] = g;
    slot_of[g] = (int32_t)slot;
    rec.kind = 1;
    rec.slot = (int32_t)slot;
    rec.evicted = v;
    out[i] = rec;
  }
  return n;
}

/*
 * Prefetch admission after a layer-step's lookup (one reading of the paper's hidden-state-guided
 * residency: experts the router ranks just below the top k are likely needed by the next token).
 * admit: the global ids to bring in, ascending. pinned: the layer-step's needed ids, ascending.
 * For each admitted id g in ascending order: if resident, nothing happens (no record). Otherwise
 * g takes the lowest free slot, else the resident v with the smallest (last_use[v], v) that is
 * neither pinned nor admitted in this call; the record has kind 2. If no slot is available the
 * remaining ids are not admitted. Admitted ids get last_use = clock.
 *
 * Returns the number of records written to out.
 */
int32_t orc_lru_admit(int64_t cap, int32_t* slot_of, int32_t* gid_of, int64_t* last_use, int64_t clock,
                      const int32_t* pinned, int32_t npinned, const int32_t* admit, int32_t nadmit, int32_t n_experts,
                      int32_t step, orc_rec* out) {
  int32_t n = 0;
  for (int32_t i = 0; i < nadmit; i++) {
    int32_t g = admit[i];
    if (slot_of[g] >= 0) continue;
    int64_t slot = -1;
    for (int64_t s = 0; s < cap; s++) {
      if (gid_of[s] < 0) {
        slot = s;
        break;
      }
    }
    int32_t victim = -1;
    if (slot < 0) {
      for (int64_t s = 0; s < cap; s++) {
        int32_t v = gid_of[s];
        if (v < 0 || in_sorted(pinned, npinned, v) || in_sorted(admit, nadmit, v)) continue;
        if (victim < 0 || last_use[v] < last_use[victim] || (last_use[v] == last_use[victim] && v < victim)) {
          victim = v;
          slot = s;
        }
      }
      if (victim < 0) break;
      slot_of[victim] = -1;
    }
    gid_of[slot] = g;
    slot_of[g] = (int32_t)slot;
    last_use[g] = clock;
    orc_rec rec;
    rec.step = step;
    rec.layer = g / n_experts;
    rec.expert = g % n_experts;
    rec.kind = 2;
    rec.slot = (int32_t)slot;
    rec.evicted = victim;
    out[n++] = rec;
  }
  return n;
}

/*
 * One layer-step under router-guided replacement (one reading of the paper's residency decisions
 * that use information produced during execution, Sec. 3, with the routing result of Fig. 1 as
 * that information). rank[gid]: the expert's rank in its layer's most recent routing (0 = highest
 * logit), n_experts for a layer not routed yet; the caller refreshes the layer's ranks before the
 * call. For each needed gid in ascending order: if resident, a hit. Otherwise the lowest free
 * slot, else the slot of the resident v outside `needed` with the largest rank[v], ties to the
 * larger last_use[v] (the more recent use), then to the lower v. Afterwards last_use[x] = clock
 * for every needed x.
 *
 * Returns the number of records, or -1 if no victim exists (cap < |needed|).
 */
int32_t orc_guided_step(int64_t cap, int32_t* slot_of, int32_t* gid_of, int64_t* last_use, const int32_t* rank,
                        int64_t clock, const int32_t* needed, int32_t n, int32_t n_experts, int32_t step,
                        orc_rec* out) {
  for (int32_t i = 0; i < n; i++) {
    int32_t g = needed[i];
    orc_rec rec;
    rec.step = step;
    rec.layer = g / n_experts;
    rec.expert = g % n_experts;
    rec.evicted = -1;
    if (slot_of[g] >= 0) {
      rec.kind = 0;
      rec.slot = slot_of[g];
      out[i] = rec;
      continue;
    }
    int64_t slot = -1;
    for (int64_t s = 0; s < cap; s++) {
      if (gid_of[s] < 0) {
        slot = s;
        break;
      }
    }
    if (slot < 0) {
      int32_t victim = -1;
      for (int64_t s = 0; s < cap; s++) {
        int32_t v = gid_of[s];
        if (v < 0 || in_sorted(needed, n, v)) continue;
        int better = 0;
        if (victim < 0)
          better = 1;
        else if (rank[v] != rank[victim])
          better = rank[v] > rank[victim];
        else if (last_use[v] != last_use[victim])
          better = last_use[v] > last_use[victim];
        else
          better = v < victim;
        if (better) {
          victim = v;
          slot = s;
        }
      }
      if (victim < 0) return -1;
      slot_of[victim] = -1;
      rec.evicted = victim;
    }
    gid_of[slot] = g;
    slot_of[g] = (int32_t)slot;
    rec.kind = 1;
    rec.slot = (int32_t)slot;
    out[i] = rec;
  }
  for (int32_t i = 0; i < n; i++) last_use[needed[i]] = clock;
  return n;
}

/* ---------------------------------------------------------------------------------------------
 * The decoder block around the MoE layer (a chained stack: attention with a KV cache, then the
 * MoE layer, each on a residual stream). The paper ran a whole MoE decoder with a 4096-token
 * context; it prints no architecture, so these follow a Qwen3-MoE-class block.
 * ------------------------------------------------------------------------------------------- */

/* RMSNorm: out_i = w_i * x_i / sqrt(mean_j x_j^2 + eps). */
void orc_rmsnorm(const double* x, const double* w, int32_t n, double eps, double* out) {
  double ss = 0.0;
  for (int32_t i = 0; i < n; i++) ss += x[i] * x[i];
  const double r = 1.0 / sqrt(ss / (double)n + eps);
  for (int32_t i = 0; i < n; i++) out[i] = w[i] * (x[i] * r);
}

/* Rotary position embedding of one head vector of even length D at position pos, pairing
 * element i with element i + D/2 (rotate-half layout): with a_i = pos * theta^(-2i/D),
 *   out_i       = x_i cos a_i - x_{i+D/2} sin a_i
 *   out_{i+D/2} = x_{i+D/2} cos a_i + x_i sin a_i            for 0 <= i < D/2. */
void orc_rope(const double* x, int32_t D, int64_t pos, double theta, double* out) {
  const int32_t h = D / 2;
  for (int32_t i = 0; i < h; i++) {
    const double a = (double)pos * pow(theta, -2.0 * (double)i / (double)D);
    const double c = cos(a), s = sin(a);
    const double x0 = x[i], x1 = x[i + h];
    out[i] = x0 * c - x1 * s;
    out[i + h] = x1 * c + x0 * s;
  }
}

/* Grouped-query attention of one query token over T cached positions.
 * q [Hq x D]; K, V [Hkv x Tmax x D] (position j of kv head g at (g * Tmax + j) * D); Hq a multiple
 * of Hkv, query head h reads kv head h / (Hq / Hkv). s_j = (q_h . K_gj) / sqrt(D) for j < T;
 * w = softmax(s) (maximum subtracted); out_h = sum_j w_j V_gj. scratch holds T doubles. */
void orc_attend(const double* q, const double* K, const double* V, int32_t Hq, int32_t Hkv, int64_t T, int64_t Tmax,
                int32_t D, double* out, double* scratch) {
  const int32_t group = Hq / Hkv;
  const double scale = 1.0 / sqrt((double)D);
  for (int32_t h = 0; h < Hq; h++) {
    const int32_t g = h / group;
    const double* qh = q + (int64_t)h * D;
    double m = -INFINITY;
    for (int64_t j = 0; j < T; j++) {
      const double* kj = K + ((int64_t)g * Tmax + j) * D;
      double acc = 0.0;
      for (int32_t i = 0; i < D; i++) acc += qh[i] * kj[i];
      scratch[j] = acc * scale;
      if (scratch[j] > m) m = scratch[j];
    }
    double tot = 0.0;
    for (int64_t j = 0; j < T; j++) {
      scratch[j] = exp(scratch[j] - m);
      tot += scratch[j];
    }
    double* oh = out + (int64_t)h * D;
    for (int32_t i = 0; i < D; i++) oh[i] = 0.0;
    for (int64_t j = 0; j < T; j++) {
      const double wj = scratch[j] / tot;
      const double* vj = V + ((int64_t)g * Tmax + j) * D;
      for (int32_t i = 0; i < D; i++) oh[i] += wj * vj[i];
    }
  }
}
