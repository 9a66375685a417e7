"""Full-size high-resolution batch (8 images, 2304 and 4096 visual tokens, 128 text
tokens, 4 layers) against the oracle, plus its compaction (GPU)."""
import numpy as np
import pytest
import torch

from oracle import e2s_oracle as orc
from tests import parity
from tests.gpu_helpers import config_inputs, config_oracle, device, run_gpu

pytestmark = pytest.mark.gpu


def test_highres_full_batch():
    inp = config_inputs(4, None, None)
    ref = config_oracle(4, None, None, "causal")
    gpu = run_gpu(inp, "causal")
    assert gpu["status"] == 0
    parity.check_floats(gpu, ref)
    parity.check_selection(gpu["keep"], gpu["q_tilde"], ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
    assert [len(k) for k in gpu["keep"]] == [253, 451] * 4


def test_qwen2vl_full_batch_compaction():
    """Ragged dynamic-resolution batch: hidden 3584 and 4 kv heads, bit-exact gather."""
    from paper_2608_23253_gb300.decision import bf16_tensor
    dev = device()
    inp = config_inputs(3, None, None, True)
    ref = orc.decide(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text, inp.grid_h, inp.grid_w,
                     inp.keep, H_kv=inp.spec.H_kv, params=orc.Params())
    gpu = run_gpu(inp, "causal")
    dec = gpu["decision"]
    dec.keep_idx.copy_(torch.as_tensor(np.concatenate(ref["keep"]).astype(np.int32), device=dev))
    L = inp.spec.L
    src_h = [inp.hidden] + [inp.k[l].reshape(inp.k.shape[1], -1) for l in range(L)] + \
            [inp.v[l].reshape(inp.v.shape[1], -1) for l in range(L)]
    src = [bf16_tensor(x, dev) for x in src_h]
    R = dec.out_rows()
    dst = [torch.empty((R, t.shape[1]), dtype=t.dtype, device=dev) for t in src]
    dec.compact(src, dst)
    torch.cuda.synchronize()
    assert dec.status() == 0
    for d_, h_ in zip(dst, src_h):
        want = orc.compact(h_, inp.n_sys, inp.n_vis, inp.n_text, ref["keep"])
        assert np.array_equal(d_.cpu().view(torch.int16).numpy().view(np.uint16), want)
