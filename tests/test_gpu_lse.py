"""Score from the pruning layer's own attention pass (GPU).

e2s_score_lse and e2s_decide_lse take every text row's log-sum-exp over its
causal prefix -- what a flash-attention forward of the layer returns per
query row; here the oracle's value (causal_row_lse, pinned on the CPU) in
float32 stands in for it -- and stream only the visual key tiles.  The scores
and the whole decision must match the oracle as e2s_score and e2s_decide do.
"""
import numpy as np
import pytest
import torch

from oracle import e2s_oracle as orc
from tests import parity
from tests.gpu_helpers import config_inputs, config_oracle, device

pytestmark = pytest.mark.gpu

# LLaVA batch 1 (<= 64 text rows: queries in both lane halves), ragged LLaVA
# (65..128 rows), Qwen2-VL GQA (two heads stacked per unit), high resolution
CASES = {"llava-b1": (1, None), "llava-ragged-b6": (2, 6), "qwen2vl-gqa-b4": (3, 4),
         "highres-b2": (4, 2)}


def _inputs(case):
    if case == "gqa-stack4":
        # 28 query / 4 kv heads, at most 32 text rows: four heads per unit
        from paper_2608_23253_gb300 import synth
        from paper_2608_23253_gb300.synth import ImageSpec
        ims = [ImageSpec(35, 24, 24, 32, 40, 3, 64), ImageSpec(3, 13, 17, 9, 12, 2, 50),
               ImageSpec(0, 30, 20, 1, 30, 3, 66)]
        return synth.make_inputs(synth.custom_spec("lse", ims, L=2, H=28, H_kv=4, cfg_id=95),
                                 with_payload=False)
    cfg, batch = CASES[case]
    return config_inputs(cfg, batch, None)


def _reference(case, inp):
    if case == "gqa-stack4":
        from tests.gpu_helpers import run_oracle
        return run_oracle(inp, "causal")
    return config_oracle(*CASES[case], None, "causal")


def _setup(case):
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    dev = device()
    inp = _inputs(case)
    lse = orc.text_row_lse(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text,
                           H_kv=inp.spec.H_kv)
    dec = Decision(Batch.from_inputs(inp, device=dev), inp.keep, e2s.params())
    q = bf16_tensor(inp.q_text, dev)
    k = bf16_tensor(inp.k, dev)
    return inp, dec, q, k, torch.as_tensor(lse.astype(np.float32), device=dev)


@pytest.mark.parametrize("case", sorted(CASES) + ["gqa-stack4"])
def test_score_lse_matches_oracle(case):
    inp, dec, q, k, lse = _setup(case)
    ref = _reference(case, inp)
    dec.score(q, k, lse=lse)
    torch.cuda.synchronize()
    assert dec.status() == 0
    parity.check_a(dec.a.cpu().numpy(), ref["a"], causal=True)


@pytest.mark.parametrize("case", sorted(CASES) + ["gqa-stack4"])
def test_decide_lse_matches_oracle(case):
    inp, dec, q, k, lse = _setup(case)
    ref = _reference(case, inp)
    dec.decide(q, k, lse=lse)
    torch.cuda.synchronize()
    assert dec.status() == 0
    gpu = {"a": dec.a.cpu().numpy(), "mass": dec.mass.cpu().numpy(),
           "fused": dec.fused.cpu().numpy(), "q": dec.q.cpu().numpy(),
           "q_tilde": dec.q_tilde.cpu().numpy(), "keep": dec.keep_lists()}
    parity.check_floats(gpu, ref)
    parity.check_selection(gpu["keep"], gpu["q_tilde"], ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
    parity.check_topk_of_own_scores(gpu["keep"], gpu["q_tilde"], inp.n_vis, inp.keep)
    for b in parity.clear_margin_images(ref, inp.n_vis, inp.keep):
        assert np.array_equal(gpu["keep"][b], ref["keep"][b])


@pytest.mark.parametrize("case", ["llava-b1", "qwen2vl-gqa-b4"])
def test_prune_lse_compaction_bit_exact(case):
    """e2s_prune_lse: the decision from the attention lse, then every output
    row is the oracle's compaction of the keep set the GPU chose, bit for bit."""
    from paper_2608_23253_gb300.decision import bf16_tensor
    cfg, batch = CASES[case]
    inp = config_inputs(cfg, batch, None, True)
    _, dec, q, k, lse = _setup(case)
    ref = config_oracle(cfg, batch, None, "causal")
    dev = device()
    L = inp.spec.L
    host = [inp.hidden] + [inp.k[l].reshape(inp.k.shape[1], -1) for l in range(L)] + \
           [inp.v[l].reshape(inp.v.shape[1], -1) for l in range(L)]
    src = [bf16_tensor(x, dev) for x in host]
    R = dec.out_rows()
    dst = [torch.full((R, t.shape[1]), -1, dtype=t.dtype, device=dev) for t in src]
    pos = torch.full((R,), -7, dtype=torch.int32, device=dev)
    dec.prune(q, k, src, dst, pos, lse=lse)
    torch.cuda.synchronize()
    assert dec.status() == 0
    keep = dec.keep_lists()
    parity.check_a(dec.a.cpu().numpy(), ref["a"], causal=True)
    parity.check_selection(keep, dec.q_tilde.cpu().numpy(), ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
    for d_, h_ in zip(dst, host):
        want = orc.compact(h_, inp.n_sys, inp.n_vis, inp.n_text, keep)
        assert np.array_equal(d_.cpu().view(torch.int16).numpy().view(np.uint16), want)
    assert np.array_equal(pos.cpu().numpy(),
                          orc.position_ids(inp.n_sys, inp.n_vis, inp.n_text, keep))
