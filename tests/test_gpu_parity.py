"""CUDA path vs the float64 oracle on every workload configuration (GPU).

All five configurations run at their full per-image shapes; configuration 4
(high-resolution, 2304 and 4096 visual tokens) is cut to two images here and
run at its full batch of eight in test_gpu_fullsize.py.
"""
import functools

import numpy as np
import pytest
import torch

from oracle import e2s_oracle as orc
from tests import parity
from paper_2608_23253_gb300 import synth
from tests.gpu_helpers import config_inputs, config_oracle, device, run_gpu, run_oracle

pytestmark = pytest.mark.gpu

CASES = [(0, None, None), (1, None, None), (1, None, 192), (1, None, 128), (2, None, None),
         (2, None, 128), (3, None, None), (4, 2, None)]


def _id(c):
    cfg, batch, keep = c
    return f"cfg{cfg}" + (f"-b{batch}" if batch else "") + (f"-k{keep}" if keep else "")


@pytest.mark.parametrize("mode", ["causal", "eq1"])
@pytest.mark.parametrize("path", ["decide", "fuse_select", "simt"])
@pytest.mark.parametrize("case", CASES, ids=_id)
def test_decision_parity(case, path, mode):
    cfg, batch, keep = case
    if path == "simt" and keep is not None:
        pytest.skip("keep budget does not affect the score kernel")
    inp = config_inputs(cfg, batch, keep)
    ref = config_oracle(cfg, batch, keep, mode)
    # decide: e2s_decide on the tensor-core score; fuse_select: tensor-core
    # e2s_score, then the cluster launch; simt: SIMT e2s_score, then the
    # separate e2s_fuse and e2s_select calls
    gpu = run_gpu(inp, mode, simt=(path == "simt"),
                  path={"decide": "decide", "fuse_select": "fuse_select",
                        "simt": "separate"}[path])
    assert gpu["status"] == 0, gpu["status"]
    parity.check_floats(gpu, ref)
    parity.check_selection(gpu["keep"], gpu["q_tilde"], ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
    parity.check_topk_of_own_scores(gpu["keep"], gpu["q_tilde"], inp.n_vis, inp.keep)
    if parity.oracle_keep_ok(ref, inp.n_vis, inp.keep):
        for b in range(inp.spec.B):
            assert np.array_equal(gpu["keep"][b], ref["keep"][b])


@pytest.mark.parametrize("keep", [192, 128, 64])
def test_compaction_bit_exact(keep):
    """Hidden states and each evidence layer's K and V, gathered from the oracle's keep set."""
    dev = device()
    inp = config_inputs(1, None, keep, True)
    ref = orc.decide(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text, inp.grid_h, inp.grid_w,
                     inp.keep, H_kv=inp.spec.H_kv, params=orc.Params())
    gpu = run_gpu(inp, "causal")
    dec = gpu["decision"]
    dec.keep_idx.copy_(torch.as_tensor(np.concatenate(ref["keep"]).astype(np.int32), device=dev))
    from paper_2608_23253_gb300.decision import bf16_tensor
    L = inp.spec.L
    hid = bf16_tensor(inp.hidden, dev)
    ks = [bf16_tensor(inp.k[l].reshape(inp.k.shape[1], -1), dev) for l in range(L)]
    vs = [bf16_tensor(inp.v[l].reshape(inp.v.shape[1], -1), dev) for l in range(L)]
    src = [hid] + ks + vs
    R = dec.out_rows()
    dst = [torch.empty((R, t.shape[1]), dtype=t.dtype, device=dev) for t in src]
    pos = torch.empty(R, dtype=torch.int32, device=dev)
    dec.compact(src, dst, pos)
    torch.cuda.synchronize()
    assert dec.status() == 0
    host = [inp.hidden] + [inp.k[l].reshape(inp.k.shape[1], -1) for l in range(L)] + \
           [inp.v[l].reshape(inp.v.shape[1], -1) for l in range(L)]
    for d_, h_ in zip(dst, host):
        want = orc.compact(h_, inp.n_sys, inp.n_vis, inp.n_text, ref["keep"])
        got = d_.cpu().view(torch.int16).numpy().view(np.uint16)
        assert np.array_equal(got, want)
    assert np.array_equal(pos.cpu().numpy(),
                          orc.position_ids(inp.n_sys, inp.n_vis, inp.n_text, ref["keep"]))
    assert R == 35 + keep + 64


def test_compaction_from_pinned_host_sources():
    """e2s_compact with the hidden states and V in page-locked host memory (read
    in place across the host link) gathers the oracle's rows bit-exactly, on a
    ragged batch, beside K from device memory."""
    dev = device()
    inp = config_inputs(2, 6, None, True)
    ref = orc.decide(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text, inp.grid_h, inp.grid_w,
                     inp.keep, H_kv=inp.spec.H_kv, params=orc.Params())
    gpu = run_gpu(inp, "causal")
    dec = gpu["decision"]
    dec.keep_idx.copy_(torch.as_tensor(np.concatenate(ref["keep"]).astype(np.int32), device=dev))
    from paper_2608_23253_gb300.decision import bf16_tensor
    L, T = inp.spec.L, inp.k.shape[1]
    host = [inp.hidden] + [inp.k[l].reshape(T, -1) for l in range(L)] + \
           [inp.v[l].reshape(T, -1) for l in range(L)]
    pinned = lambda x: torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).pin_memory()  # noqa: E731
    src = [pinned(host[0])] + [bf16_tensor(h, dev) for h in host[1:1 + L]] + \
          [pinned(h) for h in host[1 + L:]]
    R = dec.out_rows()
    dst = [torch.empty((R, t.shape[1]), dtype=torch.bfloat16, device=dev) for t in src]
    pos = torch.empty(R, dtype=torch.int32, device=dev)
    dec.compact(src, dst, pos)
    torch.cuda.synchronize()
    assert dec.status() == 0
    for d_, h_ in zip(dst, host):
        want = orc.compact(h_, inp.n_sys, inp.n_vis, inp.n_text, ref["keep"])
        assert np.array_equal(d_.cpu().view(torch.int16).numpy().view(np.uint16), want)


def test_ragged_compaction_bit_exact():
    dev = device()
    inp = config_inputs(2, 6, None, True)
    ref = orc.decide(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text, inp.grid_h, inp.grid_w,
                     inp.keep, H_kv=inp.spec.H_kv, params=orc.Params())
    gpu = run_gpu(inp, "causal")
    dec = gpu["decision"]
    dec.keep_idx.copy_(torch.as_tensor(np.concatenate(ref["keep"]).astype(np.int32), device=dev))
    from paper_2608_23253_gb300.decision import bf16_tensor
    hid = bf16_tensor(inp.hidden, dev)
    out = torch.empty((dec.out_rows(), hid.shape[1]), dtype=hid.dtype, device=dev)
    pos = torch.empty(dec.out_rows(), dtype=torch.int32, device=dev)
    dec.compact([hid], [out], pos)
    torch.cuda.synchronize()
    assert dec.status() == 0
    want = orc.compact(inp.hidden, inp.n_sys, inp.n_vis, inp.n_text, ref["keep"])
    assert np.array_equal(out.cpu().view(torch.int16).numpy().view(np.uint16), want)
    assert np.array_equal(pos.cpu().numpy(),
                          orc.position_ids(inp.n_sys, inp.n_vis, inp.n_text, ref["keep"]))


@pytest.mark.parametrize("cfg,batch", [(1, None), (2, 6), (3, 4)], ids=["cfg1", "cfg2-b6",
                                                                        "cfg3-b4"])
def test_prune_whole_step(cfg, batch):
    """e2s_prune (decide, then compaction whose fixed rows overlap the decision):
    the decision matches the oracle, and every output row is the oracle's
    compaction of the keep set the GPU chose, bit for bit."""
    inp = config_inputs(cfg, batch, None, True)
    _check_prune(inp, config_oracle(cfg, batch, None, "causal"))


def _check_prune(inp, ref):
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    dev = device()
    dec = Decision(Batch.from_inputs(inp, device=dev), inp.keep, e2s.params())
    L = inp.spec.L
    host = [inp.hidden] + [inp.k[l].reshape(inp.k.shape[1], -1) for l in range(L)] + \
           [inp.v[l].reshape(inp.v.shape[1], -1) for l in range(L)]
    src = [bf16_tensor(x, dev) for x in host]
    R = dec.out_rows()
    dst = [torch.full((R, t.shape[1]), -1, dtype=t.dtype, device=dev) for t in src]
    pos = torch.full((R,), -7, dtype=torch.int32, device=dev)
    dec.prune(bf16_tensor(inp.q_text, dev), bf16_tensor(inp.k, dev), src, dst, pos)
    torch.cuda.synchronize()
    assert dec.status() == 0
    gpu = {"a": dec.a.cpu().numpy(), "mass": dec.mass.cpu().numpy(),
           "fused": dec.fused.cpu().numpy(), "q": dec.q.cpu().numpy(),
           "q_tilde": dec.q_tilde.cpu().numpy(), "keep": dec.keep_lists()}
    parity.check_floats(gpu, ref)
    parity.check_selection(gpu["keep"], gpu["q_tilde"], ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
    parity.check_topk_of_own_scores(gpu["keep"], gpu["q_tilde"], inp.n_vis, inp.keep)
    if parity.oracle_keep_ok(ref, inp.n_vis, inp.keep):
        for b in range(inp.spec.B):
            assert np.array_equal(gpu["keep"][b], ref["keep"][b])
    for d_, h_ in zip(dst, host):
        want = orc.compact(h_, inp.n_sys, inp.n_vis, inp.n_text, gpu["keep"])
        assert np.array_equal(d_.cpu().view(torch.int16).numpy().view(np.uint16), want)
    assert np.array_equal(pos.cpu().numpy(),
                          orc.position_ids(inp.n_sys, inp.n_vis, inp.n_text, gpu["keep"]))


# Sec. 4.5 evaluates Qwen2-VL-7B at visual-token reductions of 66.7 % and
# 77.8 % (K = N_V / 3 and 2 N_V / 9 per image).  Its dynamic resolution gives
# merged-patch grids of any shape, most of them not divisible by G = 4.
DYNRES = {"r66.7": 1 / 3, "r77.8": 2 / 9}


@functools.lru_cache(maxsize=None)
def _dynres(ratio: str):
    inp = synth.make_inputs(synth.config_spec(3, keep_ratio=DYNRES[ratio], dynamic_grids=True),
                            with_payload=True)
    return inp, run_oracle(inp, "causal")


@pytest.mark.parametrize("path", ["prune", "fuse_select", "separate"])
@pytest.mark.parametrize("ratio", sorted(DYNRES))
def test_qwen2vl_dynamic_resolution(ratio, path):
    inp, ref = _dynres(ratio)
    assert sum(int(h) % 4 != 0 or int(w) % 4 != 0 for h, w in zip(inp.grid_h, inp.grid_w)) >= 8
    if path == "prune":
        _check_prune(inp, ref)
        return
    gpu = run_gpu(inp, "causal", path=path)
    assert gpu["status"] == 0, gpu["status"]
    parity.check_floats(gpu, ref)
    parity.check_selection(gpu["keep"], gpu["q_tilde"], ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
    parity.check_topk_of_own_scores(gpu["keep"], gpu["q_tilde"], inp.n_vis, inp.keep)
    for b in parity.clear_margin_images(ref, inp.n_vis, inp.keep):
        assert np.array_equal(gpu["keep"][b], ref["keep"][b])
