"""The oracle's pins catch plausible mistakes: each case builds the oracle's C source with one
deliberate mistake planted in it (a flipped tie-break, a dropped term, a wrong index or sign), loads
that build in place of the real one, and checks that the pins named for it fail. CPU only; the real
build is restored after every case."""
import os

import pytest

import oracle
from tests import test_oracle_decoder as DEC
from tests import test_oracle_expert as EXP
from tests import test_oracle_guided as GUI
from tests import test_oracle_lru as LRU
from tests import test_oracle_prefetch as PRE
from tests import test_oracle_rotary as ROT
from tests import test_oracle_router as RTR

SRC = os.path.join(os.path.dirname(oracle.__file__), "moe_oracle.c")

# name: (text in the source, its replacement, which occurrence (0 = first), pins that must fail)
MUTATIONS = {
    "top-k ties to the higher id": (
        "if (best < 0 || z[e] > z[best]) best = e;", "if (best < 0 || z[e] >= z[best]) best = e;", 0,
        [RTR.test_ties_break_toward_lower_id]),
    "gates renormalised over the wrong experts": (
        "for (int32_t r = 0; r < k; r++) s += p[idx[r]];", "for (int32_t r = 0; r < k; r++) s += p[r];", 0,
        [lambda: RTR.test_renorm_gates_equal_softmax_over_selected_logits(0)]),
    "softmax without the maximum subtracted": (
        "p[e] = exp(z[e] - m);", "p[e] = exp(z[e]);", 0, [RTR.test_softmax_shift_invariance_and_no_overflow]),
    "silu dropped from the expert": (
        "u[i] = a[i] * sig * b[i];", "u[i] = a[i] * b[i];", 0, [EXP.test_expert_matches_python_loops]),
    "combine drops the last rank": (
        "for (int32_t r = 0; r < k; r++) acc += gate[r] * y[(int64_t)r * d + i];",
        "for (int32_t r = 0; r < k - 1; r++) acc += gate[r] * y[(int64_t)r * d + i];", 0,
        [EXP.test_combine_is_gate_weighted_sum_in_rank_order]),
    "int4 nibbles swapped": (
        "int nib = (c % 2 == 0) ? (byte & 0xF) : (byte >> 4);", "int nib = (c % 2 == 0) ? (byte >> 4) : (byte & 0xF);",
        0, [EXP.test_widen_int4_hand_packed]),
    "LRU evicts the most recent": (
        "last_use[v] < last_use[victim] || (last_use[v] == last_use[victim] && v < victim)",
        "last_use[v] > last_use[victim] || (last_use[v] == last_use[victim] && v < victim)", 0,
        [LRU.test_hand_simulated_four_slot_trace]),
    "LRU ties to the higher id": (
        "last_use[v] < last_use[victim] || (last_use[v] == last_use[victim] && v < victim)",
        "last_use[v] < last_use[victim] || (last_use[v] == last_use[victim] && v > victim)", 0,
        [LRU.test_hand_simulated_four_slot_trace]),
    "rotary without reverse rotation": (
        "if (prior[s] == g && (gid_of[s] < 0 || !in_sorted(needed, n, gid_of[s]))) {",
        "if (0 && prior[s] == g) {", 0, [ROT.test_hand_simulated_four_slot_trace]),
    "admission may evict another candidate": (
        "if (v < 0 || in_sorted(pinned, npinned, v) || in_sorted(admit, nadmit, v)) continue;",
        "if (v < 0 || in_sorted(pinned, npinned, v)) continue;", 0,
        [PRE.test_admitted_experts_are_protected_from_each_other]),
    "guided ties to the older use": (
        "better = last_use[v] > last_use[victim];", "better = last_use[v] < last_use[victim];", 0,
        [lambda: GUI.test_hand_simulated_traces("B")]),
    "guided evicts the best rank": (
        "better = rank[v] > rank[victim];", "better = rank[v] < rank[victim];", 0,
        [lambda: GUI.test_hand_simulated_traces("A")]),
    "RMSNorm without eps": (
        "const double r = 1.0 / sqrt(ss / (double)n + eps);", "const double r = 1.0 / sqrt(ss / (double)n);", 0,
        [DEC.test_rmsnorm_closed_form_and_scale_invariance]),
    "rotary embedding with a wrong sign": (
        "out[i + h] = x1 * c + x0 * s;", "out[i + h] = x1 * c - x0 * s;", 0,
        [lambda: DEC.test_rope_matches_complex_rotation(17)]),
    "attention without 1/sqrt(D)": (
        "scratch[j] = acc * scale;", "scratch[j] = acc;", 0, [lambda: DEC.test_attention_matches_loops(4, 2, 5)]),
    "query heads read the wrong kv head": (
        "const int32_t g = h / group;", "const int32_t g = h % Hkv;", 0,
        [lambda: DEC.test_attention_matches_loops(4, 2, 5), DEC.test_grouped_query_equals_multi_head_with_repeated_kv]),
}


def _mutated_source(text, repl, occurrence):
    src = open(SRC).read()
    pos = -1
    for _ in range(occurrence + 1):
        pos = src.find(text, pos + 1)
        assert pos >= 0, f"mutation target not found: {text}"
    return src[:pos] + repl + src[pos + len(text):]


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_pins_catch_the_planted_mistake(name, tmp_path):
    text, repl, occ, pins = MUTATIONS[name]
    src = tmp_path / "moe_oracle_mutant.c"
    src.write_text(_mutated_source(text, repl, occ))
    so = oracle.compile_source(str(src), str(tmp_path / "liboracle_mutant.so"))
    real = oracle.lib()
    try:
        oracle._lib = oracle.load_library(so)
        caught = 0
        for pin in pins:
            try:
                pin()
            except Exception:  # any failure of the pin counts (an assertion, or an impossible state)
                caught += 1
        assert caught > 0, f"no pin caught: {name}"
    finally:
        oracle._lib = real
    RTR.test_ties_break_toward_lower_id()  # the real build is back


def _decoder_mutants():
    """Mistakes in the decoder stack's Python orchestration, as replacement methods."""
    import numpy as np

    from oracle import decoder as D

    orig_attention = D.DecoderOracle.attention

    def rope_position_off_by_one(self, l, x):
        orig = D.rope
        D.rope = lambda v, pos, theta: orig(v, pos + 1, theta)
        try:
            return orig_attention(self, l, x)
        finally:
            D.rope = orig

    def value_not_cached(self, l, x):
        out = orig_attention(self, l, x)
        self.V[l][:, self.pos] = 0.0  # the new position's value row is lost for later tokens
        return out

    def wrong_norm_weights(self, l, x):
        w = self.attn_w[l]
        saved = w["norm_in"]
        w["norm_in"] = w["norm_post"]
        try:
            return orig_attention(self, l, x)
        finally:
            w["norm_in"] = saved

    def no_qk_norm(self, l, x):
        orig = D.rmsnorm
        calls = {"n": 0}

        def rms(v, w, eps):
            calls["n"] += 1
            return orig(v, w, eps) if calls["n"] == 1 else np.asarray(v, dtype=np.float64)

        D.rmsnorm = rms
        try:
            return orig_attention(self, l, x)
        finally:
            D.rmsnorm = orig

    return {"rotary position off by one": rope_position_off_by_one, "value row not cached": value_not_cached,
            "input norm uses the post-attention weights": wrong_norm_weights, "no q/k norm": no_qk_norm}


@pytest.mark.parametrize("name", list(_decoder_mutants()))
def test_decoder_pin_catches_the_planted_mistake(name, monkeypatch):
    from oracle import decoder as D

    monkeypatch.setattr(D.DecoderOracle, "attention", _decoder_mutants()[name])
    with pytest.raises(Exception):
        DEC.test_incremental_decode_equals_the_matrix_form()
