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


def _setup(case):
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    cfg, batch = CASES[case]
    dev = device()
    inp = config_inputs(cfg, batch, None)
    lse = orc.text_row_lse(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text,
                           H_kv=inp.spec.H_kv)
    dec = Decision(Batch.from_inputs(inp, device=dev), inp.keep, e2s.params())
    q = bf16_tensor(inp.q_text, dev)
    k = bf16_tensor(inp.k, dev)
    return inp, dec, q, k, torch.as_tensor(lse.astype(np.float32), device=dev)


@pytest.mark.parametrize("case", sorted(CASES))
def test_score_lse_matches_oracle(case):
    inp, dec, q, k, lse = _setup(case)
    ref = config_oracle(*CASES[case], None, "causal")
    dec.score(q, k, lse=lse)
    torch.cuda.synchronize()
    assert dec.status() == 0
    parity.assert_close("a", dec.a.cpu().numpy(), ref["a"])


@pytest.mark.parametrize("case", sorted(CASES))
def test_decide_lse_matches_oracle(case):
    inp, dec, q, k, lse = _setup(case)
    ref = config_oracle(*CASES[case], None, "causal")
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
