"""The GPU parity bound on the score a can fail (CPU only).

At the LLaVA shapes a causal-probability score is about 1/N_V per token, the
same size as the absolute tolerance of 1e-3, so the absolute check alone
passes a score with a dropped text row or a causal mask one key short.  The
elementwise relative bound of tests/parity.py must reject both mistakes on
the seeded tiny and batch-1 LLaVA inputs, and must accept the oracle's own
values perturbed by a relative 1e-5 (the size of the GPU's float32 error).
"""
import numpy as np
import pytest

from oracle import e2s_oracle as orc
from paper_2608_23253_gb300 import synth
from tests import parity


def _scores(cfg):
    """a [L, H, N_V] of image 0 exactly, with one text row dropped, and with
    each text row's own key masked ('<' instead of '<=' in the causal mask)."""
    inp = synth.make_inputs(synth.config_spec(cfg), with_payload=False)
    S, NV, NT = int(inp.n_sys[0]), int(inp.n_vis[0]), int(inp.n_text[0])
    L, _, H, d = inp.q_text.shape
    good, drop, mask = (np.zeros((L, H, NV)) for _ in range(3))
    for l in range(L):
        for h in range(H):
            Q = orc.widen_bf16(inp.q_text[l, :NT, h])
            K = orc.widen_bf16(inp.k[l, :S + NV + NT, h])
            good[l, h] = orc.score_causal_prob(Q, K, S, NV)
            drop[l, h] = orc.score_causal_prob(Q[:-1], K[:-1], S, NV)
            logits = Q @ K.T / np.sqrt(d)
            pos = S + NV + np.arange(NT)
            vis = np.arange(K.shape[0])[None, :] < pos[:, None]
            z = np.where(vis, logits, -np.inf)
            e = np.where(vis, np.exp(z - z.max(axis=1, keepdims=True)), 0.0)
            mask[l, h] = (e / e.sum(axis=1, keepdims=True))[:, S:S + NV].mean(axis=0)
    return good, drop, mask


@pytest.mark.parametrize("cfg", [0, 1])
def test_relative_bound_rejects_plausible_score_bugs(cfg):
    good, drop, mask = _scores(cfg)
    parity.check_a(good * (1 + 1e-5), good, causal=True)
    for bad in (drop, mask):
        parity.assert_close("a", bad, good)           # the absolute bound alone is blind
        with pytest.raises(AssertionError):
            parity.check_a(bad, good, causal=True)


def test_check_floats_applies_the_relative_bound_to_causal_scores():
    good, drop, _ = _scores(0)
    L, H, N = good.shape
    ref = {"a": good, "fused": np.zeros((N, 3)), "K": np.zeros(N), "q": np.zeros(N),
           "score_mode": orc.SCORE_CAUSAL_PROB}
    gpu = {"a": drop, "fused": np.zeros((N, 4)), "q": np.zeros(N)}
    with pytest.raises(AssertionError):
        parity.check_floats(gpu, ref, mass=False)
    parity.check_floats(dict(gpu, a=good), ref, mass=False)
    # EQ1 scores (logit means, any sign) keep the absolute bound only
    parity.check_floats(dict(gpu, a=good - 0.5e-3), dict(ref, score_mode=orc.SCORE_EQ1),
                        mass=False)
