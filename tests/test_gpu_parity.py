"""CUDA path vs the float64 oracle on every workload configuration (GPU).

All five configurations run at their full per-image shapes; configuration 4
(high-resolution, 2304 and 4096 visual tokens) is cut to two images here and
run at its full batch of eight in test_gpu_fullsize.py.
"""
import numpy as np
import pytest
import torch

from oracle import e2s_oracle as orc
from tests import parity
from tests.gpu_helpers import config_inputs, config_oracle, device, run_gpu

pytestmark = pytest.mark.gpu

CASES = [(0, None, None), (1, None, None), (1, None, 192), (1, None, 128), (2, None, None),
         (2, None, 128), (3, None, None), (4, 2, None)]


def _id(c):
    cfg, batch, keep = c
    return f"cfg{cfg}" + (f"-b{batch}" if batch else "") + (f"-k{keep}" if keep else "")


@pytest.mark.parametrize("mode", ["causal", "eq1"])
@pytest.mark.parametrize("path", ["tc", "simt"])
@pytest.mark.parametrize("case", CASES, ids=_id)
def test_decision_parity(case, path, mode):
    cfg, batch, keep = case
    if path == "simt" and keep is not None:
        pytest.skip("keep budget does not affect the score kernel")
    inp = config_inputs(cfg, batch, keep)
    ref = config_oracle(cfg, batch, keep, mode)
    gpu = run_gpu(inp, mode, simt=(path == "simt"))
    assert gpu["status"] == 0, gpu["status"]
    parity.check_floats(gpu, ref)
    parity.check_selection(gpu["keep"], gpu["q_tilde"], ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
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
