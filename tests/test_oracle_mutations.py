"""Planted mistakes in the oracle must trip its pins (CPU only).

Each test patches one oracle step with a plausible error (a dropped term, a
wrong sign, an off-by-one mask, a transposed axis) and checks that the pin
written for that step rejects it.  This shows the pins are not vacuous.
"""
import json
import math
import os

import numpy as np
import pytest

from oracle import ds_generic as ds
from oracle import e2s_oracle as orc
from tests.conftest import GOLDEN


def test_mask_off_by_one_is_caught(monkeypatch):
    def bad_rows(Q, K_all, first_text_pos):
        d = Q.shape[1]
        logits = Q @ K_all.T / np.sqrt(d)
        pos = first_text_pos + np.arange(Q.shape[0])
        visible = np.arange(K_all.shape[0])[None, :] < pos[:, None]     # '<' instead of '<='
        z = np.where(visible, logits, -np.inf)
        e = np.where(visible, np.exp(z - z.max(axis=1, keepdims=True)), 0.0)
        return e / e.sum(axis=1, keepdims=True)
    r = np.random.default_rng(1)
    Q, K = r.normal(size=(1, 8)), r.normal(size=(9, 8))
    from scipy.special import softmax
    want = softmax(K @ Q[0] / math.sqrt(8))
    assert np.allclose(orc.causal_attention_rows(Q, K, 8)[0], want)
    assert not np.allclose(bad_rows(Q, K, 8)[0], want)


def test_transposed_mean_axis_is_caught():
    r = np.random.default_rng(2)
    Q, K = r.normal(size=(4, 4)), r.normal(size=(4, 4))
    good = orc.score_eq1(Q, K)
    bad = (Q @ K.T / 2.0).mean(axis=1)
    alt = K @ Q.mean(axis=0) / 2.0
    assert np.allclose(good, alt) and not np.allclose(bad, alt)


def test_clarity_sign_error_is_caught():
    g = json.load(open(os.path.join(GOLDEN, "head_support_example.json")))
    p = np.array(g["cases"][1]["p"])[:, None]
    H = 4
    p_bar = p.mean(axis=0)
    bad_clarity = (2.0 / H) * np.abs((p + 0.5).sum(axis=0))
    consistency = 1.0 - (2.0 / H) * np.abs(p - p_bar).sum(axis=0)
    assert (bad_clarity * consistency)[0] != pytest.approx(g["cases"][1]["rho"], abs=1e-6)


def test_dropped_term_in_eq14_is_caught():
    r = np.random.default_rng(3)
    A, B = r.dirichlet([1, 1, 1]), r.dirichlet([1, 1, 1])
    K = A[0] * B[1] + A[1] * B[0]
    bad_I = (A[0] * B[0] + A[0] * B[2]) / (1 - K)            # m~(Theta) m(I) dropped
    g = ds.combine({frozenset("I"): A[0], frozenset("U"): A[1], frozenset("IU"): A[2]},
                   {frozenset("I"): B[0], frozenset("U"): B[1], frozenset("IU"): B[2]})
    assert orc.dempster_combine(A[None], B[None])[0][0, 0] == pytest.approx(g[frozenset("I")])
    assert bad_I != pytest.approx(g[frozenset("I")], abs=1e-9)


def test_wrong_conflict_in_priority_is_caught():
    g = json.load(open(os.path.join(GOLDEN, "three_layer_example.json")))
    S = np.array(g["scores_by_layer"])
    masses = np.stack([orc.layer_mass(np.ones(3), S[l]) for l in range(3)])
    # cumulative conflict instead of the latest one
    f = masses[0]
    cum = np.zeros(3)
    for l in (1, 2):
        f, K = orc.dempster_combine(f, masses[l])
        cum = 1 - (1 - cum) * (1 - K)
    bad_q = 1 - (1 - orc.plausibility(f)) * (1 - cum)
    assert not np.allclose(bad_q, g["hand_fusion"]["q"], atol=1e-3)


def test_topk_tie_break_by_higher_index_is_caught():
    q = np.array([0.5, 0.7, 0.5, 0.5])
    idx = np.arange(4)
    bad = np.sort(np.lexsort((-idx, -q))[:2])
    assert orc.topk(q, 2).tolist() == [0, 1]
    assert bad.tolist() != [0, 1]


def test_lse_prefix_off_by_one_is_caught():
    """A normaliser that stops one key short of the row's own position fails
    the library logsumexp pin of causal_row_lse."""
    from scipy.special import logsumexp
    r = np.random.default_rng(13)
    Q, K = r.normal(size=(3, 8)), r.normal(size=(10, 8))
    logits = Q @ K.T / math.sqrt(8)
    want = np.array([logsumexp(logits[t, :4 + t + 1]) for t in range(3)])
    bad = np.array([logsumexp(logits[t, :4 + t]) for t in range(3)])
    assert np.allclose(orc.causal_row_lse(Q, K, 4), want, atol=1e-12)
    assert not np.allclose(bad, want, atol=1e-6)


def test_attention_mask_including_the_next_key_is_caught():
    """An attention mask one key too wide ('<= p + 1') fails the identity-value pin."""
    from scipy.special import softmax
    r = np.random.default_rng(43)
    T, d = 6, 4
    Q, K = r.normal(size=(T, d)), r.normal(size=(T, d))
    logits = Q @ K.T / 2.0
    vis = np.arange(T)[None, :] <= np.arange(T)[:, None] + 1
    z = np.where(vis, logits, -np.inf)
    bad = np.exp(z - z.max(axis=1, keepdims=True))
    bad = bad / bad.sum(axis=1, keepdims=True)
    good, _ = orc.causal_attention_output(Q, K, np.eye(T))
    assert np.allclose(good[2, :3], softmax(logits[2, :3]))
    assert not np.allclose(bad[2, :3], softmax(logits[2, :3]))
