"""The C-ABI library: loads, exports every declared symbol, validates on the host.

No GPU: only calls that fail host-side validation (before any CUDA call) or
that touch no device are made here.
"""
import ctypes
import os
import re

import pytest

from tests.conftest import ROOT


def _lib():
    path = os.path.join(ROOT, "paper_2608_23253_gb300", "libe2s.so")
    if not os.path.exists(path):
        from paper_2608_23253_gb300 import build_lib
        build_lib.build()
    from paper_2608_23253_gb300 import e2s
    return e2s


def _declared():
    names = set()
    hdr_dir = os.path.join(ROOT, "include")
    for f in os.listdir(hdr_dir):
        if f.endswith(".h"):
            src = open(os.path.join(hdr_dir, f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(e2s_[a-z_0-9]+)\s*\(", src))
    return names


def test_exports_every_declared_symbol():
    e2s = _lib()
    declared = _declared()
    assert declared >= {"e2s_score", "e2s_fuse", "e2s_select", "e2s_compact"}
    for name in declared:
        assert hasattr(e2s.lib, name), name
    assert set(e2s.EXPORTED) == declared


def _layout(e2s, **kw):
    fake = 0x1000   # never dereferenced: every case below fails validation first
    base = dict(B=1, L=2, H=32, H_kv=32, d=128, tok_off=fake, n_sys=fake, n_vis=fake,
                n_text=fake, grid_h=fake, grid_w=fake, vis_off=fake, text_off=fake,
                max_T=643, max_vis=576, max_text=32, sum_T=643, sum_vis=576, sum_text=32)
    base.update(kw)
    return e2s.e2s_layout(**base)


def test_workspace_size_and_versions():
    e2s = _lib()
    lay = _layout(e2s)
    n = e2s.e2s_workspace_size(lay, e2s.params())
    # status word, one float4 per (image, layer, head), 64 cell keys + a counter per image
    assert n == 256 + ((1 * 2 * 32 * 16 + 255) // 256) * 256 + ((1 * 129 * 4 + 255) // 256) * 256
    assert e2s.e2s_workspace_size(_layout(e2s, d=64), e2s.params()) == 0
    assert e2s.e2s_version() == 103
    assert e2s.e2s_status_string(e2s.E2S_ERR_TIMEOUT) == "E2S_ERR_TIMEOUT"
    assert e2s.e2s_status_string(99) == "E2S_ERR_UNKNOWN"


@pytest.mark.parametrize("case,want", [
    ("null_layout", "E2S_ERR_INVALID_ARG"),
    ("bad_d", "E2S_ERR_UNSUPPORTED"),
    ("gqa_mismatch", "E2S_ERR_SHAPE"),
    ("null_params", "E2S_ERR_INVALID_ARG"),
    ("bad_mode", "E2S_ERR_INVALID_ARG"),
    ("eq1_renorm", "E2S_ERR_UNSUPPORTED"),
    ("bad_G", "E2S_ERR_INVALID_ARG"),
    ("bad_lambda", "E2S_ERR_INVALID_ARG"),
    ("no_ws", "E2S_ERR_WORKSPACE"),
    ("small_ws", "E2S_ERR_WORKSPACE"),
    ("misaligned_ws", "E2S_ERR_WORKSPACE"),
    ("short_stride", "E2S_ERR_SHAPE"),
    ("misaligned_q", "E2S_ERR_ALIGNMENT"),
    ("too_many_text", "E2S_ERR_UNSUPPORTED"),
    ("unknown_flag", "E2S_ERR_INVALID_ARG"),
])
def test_score_host_validation(case, want):
    e2s = _lib()
    lay = _layout(e2s)
    par = e2s.params()
    ws, wsb = 0x100000, 1 << 20
    q, k, qs, ks = 0x200000, 0x300000, 32 * 128, 32 * 128
    if case == "null_layout":
        lay = None
    elif case == "bad_d":
        lay = _layout(e2s, d=64)
    elif case == "gqa_mismatch":
        lay = _layout(e2s, H=28, H_kv=8)
    elif case == "null_params":
        par = None
    elif case == "bad_mode":
        par = e2s.params(score_mode=7)
    elif case == "eq1_renorm":
        par = e2s.params(score_mode=e2s.E2S_SCORE_EQ1, norm_mode=e2s.E2S_NORM_RENORM)
    elif case == "bad_G":
        par = e2s.params(G=0)
    elif case == "bad_lambda":
        par = e2s.params(lam=1.5)
    elif case == "no_ws":
        ws = None
    elif case == "small_ws":
        wsb = 64
    elif case == "misaligned_ws":
        ws = 0x100010
    elif case == "short_stride":
        qs = 100
    elif case == "misaligned_q":
        q = 0x200008
    elif case == "too_many_text":
        lay = _layout(e2s, max_text=300, sum_text=300, max_T=911, sum_T=911)
    elif case == "unknown_flag":
        par = e2s.params(flags=1 << 20)
    st = e2s.e2s_score(lay, par, q, qs, k, ks, 0x400000, ws, wsb, None)
    assert e2s.e2s_status_string(st) == want


@pytest.mark.parametrize("case,want", [
    ("null_lse", "E2S_ERR_INVALID_ARG"),
    ("misaligned_lse", "E2S_ERR_ALIGNMENT"),
    ("eq1", "E2S_ERR_UNSUPPORTED"),
    ("simt", "E2S_ERR_UNSUPPORTED"),
    ("misaligned_q", "E2S_ERR_ALIGNMENT"),
])
def test_score_lse_host_validation(case, want):
    """e2s_score_lse / e2s_decide_lse: the text rows' lse is required, 4-byte
    aligned, and only the causal-probability score on the tcgen05 path uses it."""
    e2s = _lib()
    lay = _layout(e2s)
    par = e2s.params()
    ws, wsb = 0x100000, 1 << 20
    q, k, qs, ks, lse = 0x200000, 0x300000, 32 * 128, 32 * 128, 0x500000
    if case == "null_lse":
        lse = None
    elif case == "misaligned_lse":
        lse = 0x500002
    elif case == "eq1":
        par = e2s.params(score_mode=e2s.E2S_SCORE_EQ1)
    elif case == "simt":
        par = e2s.params(flags=e2s.E2S_SIMT_SCORE)
    elif case == "misaligned_q":
        q = 0x200008
    st = e2s.e2s_score_lse(lay, par, q, qs, k, ks, lse, 0x400000, ws, wsb, None)
    assert e2s.e2s_status_string(st) == want
    st = e2s.e2s_decide_lse(lay, par, q, qs, k, ks, lse, None, None, 0x400000, None, 0x600000,
                            0x700000, 0x800000, 0x900000, 64, 0xA00000, None, ws, wsb, None)
    assert e2s.e2s_status_string(st) == want
    st = e2s.e2s_prune_lse(lay, par, q, qs, k, ks, lse, None, None, 0x400000, None, 0x600000,
                           0x700000, 0x800000, 0x900000, 64, 0xA00000, None, 0, [], [], [], None,
                           ws, wsb, None)
    assert e2s.e2s_status_string(st) == want


def test_compact_host_validation():
    e2s = _lib()
    lay = _layout(e2s, sum_T=643, sum_vis=576)
    ws = 0x100000
    ok_args = dict(keep_idx=0x1000, keep_off=0x2000, sum_keep=64)
    st = e2s.e2s_compact(lay, ok_args["keep_idx"], ok_args["keep_off"], 64, 1, [0x10000],
                         [0x20000], [100], None, ws, 1 << 20)
    assert st == e2s.E2S_ERR_ALIGNMENT
    st = e2s.e2s_compact(lay, 0x1000, 0x2000, 64, 40, [0x10000] * 40, [0x20000] * 40,
                         [256] * 40, None, ws, 1 << 20)
    assert st == e2s.E2S_ERR_INVALID_ARG
    st = e2s.e2s_compact(lay, 0x1000, 0x2000, 9999, 1, [0x10000], [0x20000], [256], None, ws,
                         1 << 20)
    assert st == e2s.E2S_ERR_SHAPE
    # nothing to do: no tensors and no position ids -> OK without touching the device
    st = e2s.e2s_compact(lay, 0x1000, 0x2000, 64, 0, [], [], [], None, ws, 1 << 20)
    assert st == e2s.E2S_OK


def test_select_and_fuse_host_validation():
    e2s = _lib()
    lay = _layout(e2s)
    par = e2s.params()
    ws = 0x100000
    assert e2s.e2s_select(lay, par, 0x1000, None, None, 0x2000, 64, 0x3000, None, ws,
                          1 << 20) == e2s.E2S_ERR_INVALID_ARG
    assert e2s.e2s_select(lay, par, 0x1000, None, 0x1000, 0x2000, -1, 0x3000, None, ws,
                          1 << 20) == e2s.E2S_ERR_INVALID_ARG
    assert e2s.e2s_fuse(lay, par, None, None, None, None, 0x1000, 0x2000, ws,
                        1 << 20) == e2s.E2S_ERR_INVALID_ARG
    assert e2s.e2s_fuse(lay, par, 0x1000, None, 0x1004, None, 0x1000, 0x2000, ws,
                        1 << 20) == e2s.E2S_ERR_ALIGNMENT
    assert e2s.e2s_read_status(None) == e2s.E2S_ERR_WORKSPACE


@pytest.mark.parametrize("case,want", [
    ("no_keep_count", "E2S_ERR_INVALID_ARG"),
    ("no_keep_idx", "E2S_ERR_INVALID_ARG"),
    ("no_a_out", "E2S_ERR_INVALID_ARG"),
    ("misaligned_fused", "E2S_ERR_ALIGNMENT"),
    ("small_ws", "E2S_ERR_WORKSPACE"),
    ("too_many_heads", "E2S_ERR_UNSUPPORTED"),
])
def test_decide_host_validation(case, want):
    e2s = _lib()
    lay = _layout(e2s)
    par = e2s.params()
    ws, wsb = 0x100000, 1 << 20
    a, fused, keep_count, keep_idx = 0x400000, 0x500000, 0x600000, 0x700000
    if case == "no_keep_count":
        keep_count = None
    elif case == "no_keep_idx":
        keep_idx = None
    elif case == "no_a_out":
        a = None
    elif case == "misaligned_fused":
        fused = 0x500008
    elif case == "small_ws":
        wsb = e2s.e2s_workspace_size(lay, par) - 4
    elif case == "too_many_heads":
        lay = _layout(e2s, H=512, H_kv=512)
    st = e2s.e2s_decide(lay, par, 0x200000, lay.H * 128, 0x300000, lay.H_kv * 128, None, None,
                        a, None, fused, 0x580000, keep_count, 0x680000, 64, keep_idx, None,
                        ws, wsb, None)
    assert e2s.e2s_status_string(st) == want


def test_selftest_bounded_wait_host_validation():
    e2s = _lib()
    assert e2s.e2s_selftest_bounded_wait(0, 50_000_000, None) == e2s.E2S_ERR_WORKSPACE
    assert e2s.e2s_selftest_bounded_wait(0, 50_000_000, 0x1010) == e2s.E2S_ERR_WORKSPACE
    assert e2s.e2s_selftest_bounded_wait(0, 10, 0x1000) == e2s.E2S_ERR_INVALID_ARG
    assert e2s.e2s_selftest_bounded_wait(0, 3_000_000_000, 0x1000) == e2s.E2S_ERR_INVALID_ARG


def test_attention_host_validation():
    e2s = _lib()
    lay = _layout(e2s)
    ws = 0x100000
    wsb = e2s.e2s_workspace_size(lay, e2s.params())
    fake = 0x2000
    # every call below fails host validation, so nothing is launched
    assert e2s.e2s_attention(lay, None, 4096, fake, 4096, fake, 4096, fake, 4096, None, None,
                             ws, wsb) == e2s.E2S_ERR_INVALID_ARG
    assert e2s.e2s_attention(lay, fake, 4000, fake, 4096, fake, 4096, fake, 4096, None, None,
                             ws, wsb) == e2s.E2S_ERR_SHAPE
    assert e2s.e2s_attention(lay, fake + 8, 4096, fake, 4096, fake, 4096, fake, 4096, None, None,
                             ws, wsb) == e2s.E2S_ERR_ALIGNMENT
    assert e2s.e2s_attention(_layout(e2s, max_text=129, max_T=700, sum_T=700, sum_text=129),
                             fake, 4096, fake, 4096, fake, 4096, fake, 4096, None, fake, ws,
                             wsb * 2) == e2s.E2S_ERR_UNSUPPORTED
    assert e2s.e2s_decide_attn(lay, e2s.params(score_mode=e2s.E2S_SCORE_EQ1), fake, 4096, fake,
                               4096, fake, 4096, fake, 4096, None, None, None, fake, None, fake,
                               fake, fake, fake, 0, None, None, ws, wsb) == e2s.E2S_ERR_UNSUPPORTED
