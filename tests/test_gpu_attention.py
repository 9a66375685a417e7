"""The pruning layer's attention pass with the score as a by-product (GPU).

e2s_attention computes every row's causal attention output O and row
normaliser lse for each image, layer and query head, and -- from the text
rows' final normalisers -- the decision's score a, so that no other pass
reads K for it.  Checked against the float64 oracle:
  * lse within 2e-4 (fp32 logits from bf16 inputs);
  * O within 2^-7 * sum_j p_j |v_j| + 1e-5 per element: the weights are
    rounded to bf16 before P V (as in flash-attention forwards) and O is
    returned in bf16, each a relative 2^-9 at most;
  * a with the parity bounds of every score (max abs 1e-3, relative 5e-4);
  * e2s_decide_attn's whole decision with the usual float and selection rules.
"""
import numpy as np
import pytest
import torch

from oracle import e2s_oracle as orc
from paper_2608_23253_gb300 import synth
from paper_2608_23253_gb300.synth import ImageSpec
from tests import parity
from tests.gpu_helpers import device, run_oracle

pytestmark = pytest.mark.gpu


def _cases(name):
    if name == "cfg0":
        spec = synth.config_spec(0)
        spec.hidden = 256            # draws V (and a small hidden state) as well
        return synth.make_inputs(spec)
    if name == "gqa-ragged":
        ims = [ImageSpec(35, 16, 16, 100, 20, 3, 28), ImageSpec(3, 8, 20, 128, 10, 2, 16),
               ImageSpec(35, 12, 12, 7, 12, 3, 17)]
        spec = synth.custom_spec("attn-gqa", ims, L=2, H=8, H_kv=2, hidden=256, cfg_id=96)
        return synth.make_inputs(spec)
    if name == "tiny-ragged":
        ims = [ImageSpec(0, 1, 1, 1, 1, 0, 1), ImageSpec(5, 3, 4, 9, 3, 0, 4),
               ImageSpec(2, 5, 7, 120, 6, 2, 40)]
        spec = synth.custom_spec("attn-tiny", ims, L=1, H=4, H_kv=4, hidden=128, cfg_id=95)
        return synth.make_inputs(spec)
    raise ValueError(name)


CASES = ["cfg0", "gqa-ragged", "tiny-ragged"]


def _run(inp, decide=False):
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    dev = device()
    s = inp.spec
    q_all = synth.full_queries(inp)
    batch = Batch.from_inputs(inp, device=dev)
    dec = Decision(batch, inp.keep, e2s.params())
    q, k, v = (bf16_tensor(x, dev) for x in (q_all, inp.k, inp.v))
    o = torch.full(q.shape, -1, dtype=torch.bfloat16, device=dev)
    lse = torch.full((s.L, s.H, batch.sum_T), float("nan"), dtype=torch.float32, device=dev)
    dec.a.fill_(float("nan"))
    if decide:
        dec.decide_attn(q, k, v, o, lse)
    else:
        dec.attention(q, k, v, o, lse)
    torch.cuda.synchronize()
    assert dec.status() == e2s.E2S_OK
    return q_all, dec, o.float().cpu().numpy(), lse.cpu().numpy()


@pytest.mark.parametrize("case", CASES)
def test_attention_output_lse_and_score(case):
    inp = _cases(case)
    q_all, dec, o, lse = _run(inp)
    O_ref, lse_ref = orc.attention_layer(q_all, inp.k, inp.v, inp.n_sys, inp.n_vis, inp.n_text,
                                         H_kv=inp.spec.H_kv)
    absv = np.abs(orc.widen_bf16(inp.v)).astype(np.float32)
    v_abs = synth.bf16_bits(absv)   # |v| is exact in bf16
    O_abs, _ = orc.attention_layer(q_all, inp.k, v_abs, inp.n_sys, inp.n_vis, inp.n_text,
                                   H_kv=inp.spec.H_kv)
    parity.assert_close("lse", lse, lse_ref, tol=2e-4)
    bound = 2.0 ** -7 * O_abs + 1e-5
    err = np.abs(o - O_ref)
    worst = np.unravel_index(int(np.argmax(err - bound)), err.shape)
    assert np.all(err <= bound), f"O: err {err[worst]:.3g} > bound {bound[worst]:.3g} at {worst}"
    ref = run_oracle(inp, "causal")
    parity.check_a(dec.a.cpu().numpy(), ref["a"], causal=True)


@pytest.mark.parametrize("case", CASES)
def test_decide_from_attention_matches_oracle(case):
    inp = _cases(case)
    _, dec, _, _ = _run(inp, decide=True)
    gpu = {"a": dec.a.cpu().numpy(), "mass": dec.mass.cpu().numpy(),
           "fused": dec.fused.cpu().numpy(), "q": dec.q.cpu().numpy(),
           "q_tilde": dec.q_tilde.cpu().numpy(), "keep": dec.keep_lists()}
    ref = run_oracle(inp, "causal")
    parity.check_floats(gpu, ref)
    parity.check_selection(gpu["keep"], gpu["q_tilde"], ref["q"], inp.n_vis, inp.grid_h,
                           inp.grid_w, inp.keep, 0.1, 4)
    parity.check_topk_of_own_scores(gpu["keep"], gpu["q_tilde"], inp.n_vis, inp.keep)


def test_attention_score_equals_separate_score():
    """The score read off the attention pass and e2s_score's on the same
    inputs agree to float32 rounding (both from fp32 logits)."""
    inp = _cases("cfg0")
    _, dec, _, _ = _run(inp)
    a_attn = dec.a.cpu().numpy()
    from paper_2608_23253_gb300.decision import bf16_tensor
    dec.score(bf16_tensor(inp.q_text, device()), bf16_tensor(inp.k, device()))
    torch.cuda.synchronize()
    parity.check_a(a_attn, dec.a.cpu().numpy().astype(np.float64), causal=True, rel=1e-5)


def _attention_raw(inp, dec, q, k, v, o, o_stride, lse):
    from paper_2608_23253_gb300 import e2s
    b = dec.batch
    e2s.check(e2s.e2s_attention(b.layout, q, b.H * b.d, k, b.H_kv * b.d, v, b.H_kv * b.d, o,
                                o_stride, lse, dec.a, dec.ws, dec.ws_bytes, None),
              "e2s_attention")


def test_attention_unaligned_output_rows():
    """O rows that are 16- but not 32-byte aligned (offset 16 bytes, row stride
    H*d + 8) take the 16-byte store path: the same bits as the aligned run, and
    the padding between rows untouched."""
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    inp = _cases("gqa-ragged")
    _, dec, o_ref, lse_ref = _run(inp)
    dev = device()
    s = inp.spec
    q = bf16_tensor(synth.full_queries(inp), dev)
    k, v = bf16_tensor(inp.k, dev), bf16_tensor(inp.v, dev)
    rows, width = s.L * dec.batch.sum_T, s.H * 128
    big = torch.full((rows, width + 8), 7.0, dtype=torch.bfloat16, device=dev)
    o = big[:, 8:8 + width]
    assert o.data_ptr() % 32 == 16
    lse = torch.full((s.L, s.H, dec.batch.sum_T), float("nan"), dtype=torch.float32, device=dev)
    _attention_raw(inp, dec, q, k, v, o, width + 8, lse)
    torch.cuda.synchronize()
    assert dec.status() == e2s.E2S_OK
    got = o.float().cpu().numpy().reshape(o_ref.shape)
    assert np.array_equal(got.view(np.uint32), o_ref.view(np.uint32))
    assert np.array_equal(lse.cpu().numpy(), lse_ref)
    assert bool((big[:, :8] == 7.0).all())


def test_attention_repeats_and_leaves_counter_zero():
    """The CTAs share an item counter in the workspace: 50 calls in a row give
    the same bits every time and leave workspace bytes 4..15 zero."""
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import bf16_tensor
    inp = _cases("cfg0")
    _, dec, o_ref, lse_ref = _run(inp)
    dev = device()
    s = inp.spec
    q = bf16_tensor(synth.full_queries(inp), dev)
    k, v = bf16_tensor(inp.k, dev), bf16_tensor(inp.v, dev)
    o = torch.empty_like(q)
    lse = torch.empty((s.L, s.H, dec.batch.sum_T), dtype=torch.float32, device=dev)
    a_ref = dec.a.clone()
    for _ in range(50):
        dec.attention(q, k, v, o, lse)
    torch.cuda.synchronize()
    assert dec.status() == e2s.E2S_OK
    assert np.array_equal(o.float().cpu().numpy().view(np.uint32), o_ref.view(np.uint32))
    assert np.array_equal(lse.cpu().numpy(), lse_ref)
    assert torch.equal(dec.a, a_ref)
    assert int(dec.ws[4:16].to(torch.int32).abs().sum()) == 0
