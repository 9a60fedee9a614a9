"""The C-ABI library builds, loads and exports every function include/moe.h declares (CPU only:
no compute call is made without a GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "moe.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(moe_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2605_29135_gb300 import _lib
    from paper_2605_29135_gb300.buildsys import build

    build()
    return _lib.load()


def test_header_declares_the_binding_exports():
    from paper_2605_29135_gb300 import _lib

    assert _declared() == sorted(_lib.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name
        assert isinstance(getattr(lib, name), ctypes._CFuncPtr)


def test_config_struct_layout_matches_header(lib):
    from paper_2605_29135_gb300._lib import MoeConfig, TraceRec

    # int32 x6, int32 x2, int64 x2, int32 x2, pointer, int64, int32 x5 (+ 4 bytes of tail padding)
    assert ctypes.sizeof(MoeConfig) == 6 * 4 + 2 * 4 + 2 * 8 + 2 * 4 + 8 + 8 + 5 * 4 + 4
    assert MoeConfig.lookahead.offset == 88
    assert ctypes.sizeof(TraceRec) == 24


def test_expert_and_pool_bytes_without_gpu(lib):
    import paper_2605_29135_gb300 as P

    c = P.make_config(2048, 128, 8, 768, 48, "bf16", "bf16", cap_bytes=6_000_000_000)
    assert P.expert_bytes(c) == 9_437_184
    assert P.pool_bytes(c) == 635 * 9_437_184
    c4 = P.make_config(2048, 128, 8, 768, 48, "int4", "bf16", cap_bytes=6_000_000_000)
    assert P.expert_bytes(c4) == 2_433_024
    assert P.pool_bytes(c4) == 2466 * 2_433_024
    c1 = P.make_config(256, 8, 2, 128, 1, "fp32", "fp32", cap_slots=4)
    assert P.expert_bytes(c1) == 393_216
    bad = P.make_config(250, 8, 2, 128, 1, "int4", "bf16", cap_slots=4)
    assert P.expert_bytes(bad) == -1


def test_invalid_config_is_rejected_before_touching_a_device(lib):
    import paper_2605_29135_gb300 as P

    bad = P.make_config(256, 8, 9, 128, 1, "fp32", "fp32", cap_slots=4)  # top_k > E
    h = ctypes.c_void_p()
    st = lib.moe_create(ctypes.byref(bad), ctypes.byref(h))
    assert st == -1 and not h.value
    assert b"top_k" in lib.moe_last_error(None)


def test_null_handle_calls_fail_cleanly(lib):
    assert lib.moe_decode_step(None, None, None, 1, None) == -1
    assert lib.moe_reset_residency(None) == -1
    lib.moe_destroy(None)


def test_rotary_policy_is_a_valid_configuration_for_batches(lib):
    # moe_expert_bytes answers -1 for a configuration that moe_create would reject
    import paper_2605_29135_gb300 as P

    cfg = P.make_config(256, 8, 2, 128, 1, "fp32", "fp32", cap_slots=4, max_batch=4, policy="rotary")
    assert lib.moe_expert_bytes(ctypes.byref(cfg)) > 0
    cfg = P.make_config(256, 8, 2, 128, 1, "fp32", "fp32", cap_slots=4, max_batch=4, policy="rotary",
                        schedule="host_copy_engine")
    assert lib.moe_expert_bytes(ctypes.byref(cfg)) == -1  # batches need the device schedule


@pytest.mark.parametrize("lang,std", [("c", "c99"), ("c++", "c++11")])
def test_header_compiles_as_plain_c_and_cpp(lang, std, tmp_path):
    # the boundary is a C ABI: the header must stand alone in C as well as C++
    import shutil
    import subprocess

    cc = shutil.which("gcc" if lang == "c" else "g++")
    if cc is None:
        pytest.skip("no host compiler")
    src = tmp_path / ("use.c" if lang == "c" else "use.cpp")
    src.write_text('#include "moe.h"\nint main(void) { moe_config c; (void)c; return (int)sizeof(moe_trace_rec) - 24; }\n')
    subprocess.run([cc, f"-std={std}", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I", os.path.join(ROOT, "include"),
                    "-fsyntax-only", str(src)], check=True)


def test_attention_scratch_size_and_argument_checks_without_gpu(lib):
    # splits: about 304 CTAs over the kv heads, at least 16 positions each, none empty
    assert lib.moe_attention_scratch_floats(32, 4, 128, 4095) == 32 * 76 * 130
    assert lib.moe_attention_scratch_floats(8, 2, 64, 100) == 8 * 7 * 66
    assert lib.moe_attention_scratch_floats(4, 4, 128, 1) == 4 * 1 * 130
    for args in [(32, 4, 96, 10), (32, 5, 128, 10), (48, 3, 128, 10), (4, 4, 128, 0), (64, 4, 128, 10)]:
        assert lib.moe_attention_scratch_floats(*args) == -1
    # NULL buffers are refused before any device work
    assert lib.moe_attention_decode(None, None, None, 1, 32, 4, 128, 4096, 10, None, None, 0, None) == -1
    # an unknown cache element type is refused too
    dummy = ctypes.c_void_p(16)
    assert lib.moe_attention_decode(dummy, dummy, dummy, 2, 32, 4, 128, 4096, 10, dummy, dummy, 1 << 30, None) == -1


def test_decoder_config_layout_and_argument_checks_without_gpu(lib):
    from paper_2605_29135_gb300._lib import DecoderConfig

    # int32 x4, int64, double x2
    assert ctypes.sizeof(DecoderConfig) == 4 * 4 + 8 + 2 * 8
    assert DecoderConfig.max_pos.offset == 16 and DecoderConfig.eps.offset == 24
    cfg = DecoderConfig(n_heads=32, n_kv_heads=4, head_dim=128, reserved=0, max_pos=4160, eps=1e-6, rope_theta=1e6)
    out = ctypes.c_void_p(1)
    assert lib.moe_decoder_create(None, ctypes.byref(cfg), ctypes.byref(out)) == -1
    assert out.value is None  # *out is cleared on failure
    assert b"NULL" in lib.moe_decoder_last_error(None)
    assert lib.moe_decoder_position(None) == -1
    assert lib.moe_decoder_step(None, None, None, None, None) == -1
    assert lib.moe_decoder_set_layer(None, 0, *([None] * 8)) == -1
    assert lib.moe_decoder_set_cache(None, 0, None, None, 0) == -1
    lib.moe_decoder_destroy(None)


def test_binding_argument_counts_match_the_header(lib):
    # every prototype in include/moe.h takes as many arguments as the ctypes declaration passes
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    protos = re.findall(r"\b(moe_[a-z_]+)\s*\(([^)]*)\)\s*;", src)
    assert len(protos) == len(_declared())
    for name, params in protos:
        params = " ".join(params.split())
        n = 0 if params in ("", "void") else params.count(",") + 1
        assert len(getattr(lib, name).argtypes) == n, name
