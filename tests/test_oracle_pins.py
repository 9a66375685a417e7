"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test checks one oracle step against something other than the oracle's
own formula: a worked example of the paper, a library routine in a special
case, brute force on tiny inputs, or an invariant.  No GPU.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
from scipy.special import softmax as sp_softmax

from oracle import ds_generic as ds
from oracle import e2s_oracle as orc
from tests.conftest import GOLDEN


def _rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- Eq. 1
def test_eq1_equals_mean_query_dot_key():
    """Eq. 1 is linear in Q_t: the mean of logits equals mean(Q) . K / sqrt(d)."""
    r = _rng(1)
    Q, K = r.normal(size=(7, 16)), r.normal(size=(11, 16))
    a = orc.score_eq1(Q, K)
    alt = K @ Q.mean(axis=0) / math.sqrt(16)
    np.testing.assert_allclose(a, alt, rtol=0, atol=1e-12)


def test_eq1_brute_force_loops():
    r = _rng(2)
    Q, K = r.normal(size=(3, 4)), r.normal(size=(5, 4))
    a = orc.score_eq1(Q, K)
    for n in range(5):
        s = 0.0
        for t in range(3):
            s += sum(Q[t, i] * K[n, i] for i in range(4)) / math.sqrt(4)
        assert abs(a[n] - s / 3) < 1e-12


# ------------------------------------------------------ causal-prefix score
def test_causal_rows_single_query_is_textbook_softmax():
    """N_T = 1 at the last position sees every key: a plain softmax row."""
    r = _rng(3)
    d, S, NV = 8, 3, 5
    Q, K = r.normal(size=(1, d)), r.normal(size=(S + NV + 1, d))
    P = orc.causal_attention_rows(Q, K, S + NV)
    np.testing.assert_allclose(P[0], sp_softmax(K @ Q[0] / math.sqrt(d)), atol=1e-14)
    a = orc.score_causal_prob(Q, K, S, NV)
    np.testing.assert_allclose(a, P[0, S:S + NV], atol=1e-15)


def test_causal_rows_brute_force_prefix():
    r = _rng(4)
    d, S, NV, NT = 4, 2, 3, 3
    Q, K = r.normal(size=(NT, d)), r.normal(size=(S + NV + NT, d))
    P = orc.causal_attention_rows(Q, K, S + NV)
    for t in range(NT):
        last = S + NV + t
        logits = [sum(Q[t, i] * K[j, i] for i in range(d)) / math.sqrt(d) for j in range(last + 1)]
        mx = max(logits)
        e = [math.exp(x - mx) for x in logits]
        z = sum(e)
        for j in range(S + NV + NT):
            want = e[j] / z if j <= last else 0.0
            assert abs(P[t, j] - want) < 1e-14
        assert abs(P[t].sum() - 1.0) < 1e-14
    a = orc.score_causal_prob(Q, K, S, NV)
    np.testing.assert_allclose(a, P[:, S:S + NV].mean(axis=0), atol=1e-15)


def test_causal_mask_hides_later_text_keys():
    r = _rng(5)
    d, S, NV, NT = 8, 2, 4, 3
    Q, K = r.normal(size=(NT, d)), r.normal(size=(S + NV + NT, d))
    P0 = orc.causal_attention_rows(Q, K, S + NV)
    K2 = K.copy()
    K2[S + NV + 2] += 10.0          # only text row 2 can see this key
    P1 = orc.causal_attention_rows(Q, K2, S + NV)
    np.testing.assert_allclose(P0[:2], P1[:2], atol=0)
    assert not np.allclose(P0[2], P1[2])


# ---------------------------------------------------------------- Eqs. 8-9
def test_softmax_normalisation_matches_scipy():
    a = _rng(6).normal(size=50) * 3
    np.testing.assert_allclose(orc.normalise_softmax(a), sp_softmax(a), atol=1e-15)


def test_renorm_sums_to_one_and_degenerate_is_uniform():
    a = _rng(7).uniform(size=40)
    assert abs(orc.normalise_renorm(a).sum() - 1) < 1e-14
    np.testing.assert_allclose(orc.normalise_renorm(np.zeros(5)), 0.2)


def test_average_attention_gives_half_support():
    """Sec. 4.1: r = 1/N_l gives p = 0.5 (no selection preference)."""
    for N in (1, 7, 576, 4096):
        assert orc.support(np.array([1.0 / N]), N)[0] == pytest.approx(0.5, abs=1e-15)


def test_support_range_and_monotone():
    r = np.sort(_rng(8).uniform(0, 1, size=100))
    p = orc.support(r, 576)
    assert np.all(p >= 0) and np.all(p < 1) and np.all(np.diff(p) >= 0)


# ---------------------------------------------------------------- Eqs. 10-11
def test_head_support_example_from_paper():
    g = json.load(open(os.path.join(GOLDEN, "head_support_example.json")))
    for case in g["cases"]:
        p = np.array(case["p"])[:, None]            # [H, 1]
        rho, p_bar = orc.reliability(p)
        assert p_bar[0] == pytest.approx(case["p_bar"], abs=1e-12)
        assert rho[0] == pytest.approx(case["rho"], abs=1e-12)
        m = orc.layer_mass(rho, p_bar)[0]
        np.testing.assert_allclose(m, case["mass"], atol=1e-12)
    # the consistent example is far more reliable than the conflicting one
    assert g["cases"][0]["rho"] > 100 * g["cases"][1]["rho"]


def test_reliability_special_cases():
    # every head at 0.5: no clarity, vacuous mass
    rho, _ = orc.reliability(np.full((8, 3), 0.5))
    np.testing.assert_allclose(rho, 0.0, atol=0)
    # identical heads: consistency 1, rho = 2 |p - 1/2|
    p = np.tile(np.array([0.1, 0.5, 0.95]), (6, 1))
    rho, _ = orc.reliability(p)
    np.testing.assert_allclose(rho, [0.8, 0.0, 0.9], atol=1e-14)


def test_mass_axioms_random():
    r = _rng(9)
    p = r.uniform(0, 0.999, size=(32, 1000))
    rho, p_bar = orc.reliability(p)
    assert np.all(rho >= 0) and np.all(rho <= 1)
    m = orc.layer_mass(rho, p_bar)
    assert np.all(m >= -1e-15)
    np.testing.assert_allclose(m.sum(axis=1), 1.0, atol=1e-14)


# ---------------------------------------------------------------- Eqs. 12-19
I_, U_ = "I", "U"
THETA = frozenset({I_, U_})


def _as_generic(m):
    return {frozenset({I_}): m[0], frozenset({U_}): m[1], THETA: m[2]}


def _random_masses(r, n):
    x = r.dirichlet([1.0, 1.0, 1.0], size=n)
    return x


def test_dempster_closed_form_equals_generic_rule():
    """Eqs. 13-16 equal Eqs. 3-4 enumerated over the focal sets of {I, U}."""
    r = _rng(10)
    A, B = _random_masses(r, 300), _random_masses(r, 300)
    fused, K = orc.dempster_combine(A, B)
    for i in range(300):
        g1, g2 = _as_generic(A[i]), _as_generic(B[i])
        assert K[i] == pytest.approx(ds.conflict(g1, g2), abs=1e-14)
        gm = ds.combine(g1, g2)
        for j, S in enumerate([frozenset({I_}), frozenset({U_}), THETA]):
            assert fused[i, j] == pytest.approx(gm.get(S, 0.0), abs=1e-12)
        assert ds.check_axioms(gm, tol=1e-12)
        assert orc.belief(fused[i]) == pytest.approx(ds.belief(gm, frozenset({I_})), abs=1e-12)
        assert orc.plausibility(fused[i]) == pytest.approx(
            ds.plausibility(gm, frozenset({I_})), abs=1e-12)


def test_dempster_commutative_and_associative():
    r = _rng(11)
    A, B, C = (_random_masses(r, 200) for _ in range(3))
    ab, _ = orc.dempster_combine(A, B)
    ba, _ = orc.dempster_combine(B, A)
    np.testing.assert_allclose(ab, ba, atol=1e-13)
    ab_c, _ = orc.dempster_combine(ab, C)
    bc, _ = orc.dempster_combine(B, C)
    a_bc, _ = orc.dempster_combine(A, bc)
    np.testing.assert_allclose(ab_c, a_bc, atol=1e-12)


def test_vacuous_mass_is_identity_and_total_conflict_is_vacuous():
    r = _rng(12)
    A = _random_masses(r, 50)
    vac = np.tile([0.0, 0.0, 1.0], (50, 1))
    f, K = orc.dempster_combine(A, vac)
    np.testing.assert_allclose(f, A, atol=1e-15)
    np.testing.assert_allclose(K, 0.0)
    f, K = orc.dempster_combine(np.array([[1.0, 0, 0]]), np.array([[0.0, 1, 0]]))
    np.testing.assert_allclose(f, [[0, 0, 1]])
    assert K[0] == 1.0
    assert orc.priority(orc.plausibility(f), K)[0] == 1.0


def test_three_layer_example():
    g = json.load(open(os.path.join(GOLDEN, "three_layer_example.json")))
    S = np.array(g["scores_by_layer"])
    assert S[:, 0].mean() == pytest.approx(g["printed_average_token1"], abs=0.005)
    masses = np.stack([orc.layer_mass(np.ones(3), S[l]) for l in range(3)])
    fused, K = orc.fuse_layers(masses)
    h = g["hand_fusion"]
    np.testing.assert_allclose(fused[0], h["fused_token1"], atol=1e-6)
    assert K[0] == pytest.approx(h["K_token1"], abs=1e-6)
    q = orc.priority(orc.plausibility(fused), K)
    np.testing.assert_allclose(q, h["q"], atol=h["q_tolerance"])


def test_priority_is_one_minus_unnormalised_U_numerator():
    """q = 1 - (1-Pl)(1-K) = 1 - [m~U mU + m~U mTheta + m~Theta mU] (Eqs. 15, 18, 19)."""
    r = _rng(13)
    A, B = _random_masses(r, 500), _random_masses(r, 500)
    fused, K = orc.dempster_combine(A, B)
    q = orc.priority(orc.plausibility(fused), K)
    numer = A[:, 1] * B[:, 1] + A[:, 1] * B[:, 2] + A[:, 2] * B[:, 1]
    np.testing.assert_allclose(q, 1.0 - numer, atol=1e-12)


def test_first_layer_priority_is_plausibility():
    m = _random_masses(_rng(14), 20)[None]
    fused, K = orc.fuse_layers(m)
    np.testing.assert_allclose(K, 0)
    np.testing.assert_allclose(orc.priority(orc.plausibility(fused), K), 1 - m[0, :, 1])


def test_prior_fusion_equals_longer_chain():
    """Carrying the fused state into a later call equals fusing all layers at once."""
    r = _rng(15)
    m = np.stack([_random_masses(r, 40) for _ in range(5)])
    f_all, K_all = orc.fuse_layers(m)
    f_2, _ = orc.fuse_layers(m[:2])
    f_rest, K_rest = orc.fuse_layers(m[2:], prior=f_2)
    np.testing.assert_allclose(f_all, f_rest, atol=1e-12)
    np.testing.assert_allclose(K_all, K_rest, atol=1e-12)


# ---------------------------------------------------------------- Eqs. 20-23
def test_cells_are_6x6_blocks_on_llava_grid():
    """Sec. 4.3: G = 4 on the 24 x 24 grid gives 16 cells of 6 x 6 tokens."""
    c = orc.cell_of(np.arange(576), 24, 24, 4).reshape(24, 24)
    for ci in range(4):
        for cj in range(4):
            block = c[6 * ci:6 * ci + 6, 6 * cj:6 * cj + 6]
            assert np.all(block == ci * 4 + cj)
    assert np.bincount(c.ravel()).tolist() == [36] * 16


def test_cells_cover_non_divisible_grid():
    for h, w in [(5, 7), (1, 1), (3, 2), (36, 36), (24, 32)]:
        c = orc.cell_of(np.arange(h * w), h, w, 4).reshape(h, w)
        assert c.min() >= 0 and c.max() < 16
        # cell ids are monotone along rows and columns (bands)
        assert np.all(np.diff(c // 4, axis=0) >= 0) and np.all(np.diff(c % 4, axis=1) >= 0)


def test_representative_brute_force():
    r = _rng(16)
    for trial in range(20):
        h, w = r.integers(1, 9, size=2)
        q = r.integers(0, 4, size=h * w).astype(float) / 4   # many ties
        cells = orc.cell_of(np.arange(h * w), h, w, 4)
        b = orc.representative_indicator(q, cells)
        for g in set(cells.tolist()):
            members = [n for n in range(h * w) if cells[n] == g]
            best = members[0]
            for n in members:
                if q[n] > q[best]:
                    best = n
            assert b[best] == 1.0
            assert sum(b[n] for n in members) == 1.0


def test_topk_brute_force_greedy():
    r = _rng(17)
    for trial in range(50):
        N = int(r.integers(0, 12))
        qt = r.integers(0, 5, size=N).astype(float)
        K = int(r.integers(0, N + 3))
        got = orc.topk(qt, K).tolist()
        left = list(range(N))
        chosen = []
        for _ in range(min(K, N)):
            best = left[0]
            for n in left:
                if qt[n] > qt[best]:
                    best = n
            chosen.append(best)
            left.remove(best)
        assert got == sorted(chosen)


def test_topk_edge_cases():
    q = np.array([0.3, 0.9, 0.1])
    assert orc.topk(q, 0).tolist() == []
    assert orc.topk(q, 10).tolist() == [0, 1, 2]
    assert orc.topk(np.full(5, 0.5), 2).tolist() == [0, 1]


# ---------------------------------------------------------------- whole decision
def _tiny_inputs(seed, L=2, H=4, Hkv=4, grids=((6, 6),), NT=(5,), S=3, d=16):
    r = _rng(seed)
    n_vis = [h * w for h, w in grids]
    T = [S + nv + nt for nv, nt in zip(n_vis, NT)]

    def bits(x):
        return (x.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    q = bits(r.normal(size=(L, sum(NT), H, d)) * 0.5)
    k = bits(r.normal(size=(L, sum(T), Hkv, d)) * 0.5)
    return q, k, [S] * len(grids), n_vis, list(NT), [g[0] for g in grids], [g[1] for g in grids]


def test_decide_invariants_tiny():
    q, k, ns, nv, nt, gh, gw = _tiny_inputs(20, grids=((6, 6), (4, 5)), NT=(5, 3))
    for mode in (orc.SCORE_EQ1, orc.SCORE_CAUSAL_PROB):
        out = orc.decide(q, k, ns, nv, nt, gh, gw, [7, 30], H_kv=4, params=orc.Params(score_mode=mode))
        np.testing.assert_allclose(out["mass"].sum(axis=-1), 1.0, atol=1e-12)
        np.testing.assert_allclose(out["fused"].sum(axis=-1), 1.0, atol=1e-12)
        assert np.all(out["mass"] >= -1e-15) and np.all(out["fused"] >= -1e-15)
        assert np.all((out["q"] >= 0) & (out["q"] <= 1 + 1e-12))
        assert [len(x) for x in out["keep"]] == [7, 20]
        if mode == orc.SCORE_CAUSAL_PROB:
            assert np.all(out["a"] > 0) and np.all(out["a"] < 1)


def test_no_novelty_selects_topk_of_priority():
    q, k, ns, nv, nt, gh, gw = _tiny_inputs(21)
    p = orc.Params(score_mode=orc.SCORE_CAUSAL_PROB, flags=orc.NO_NOVELTY)
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [9], H_kv=4, params=p)
    assert out["keep"][0].tolist() == orc.topk(out["q"], 9).tolist()
    np.testing.assert_allclose(out["q_tilde"], out["q"])


def test_certain_single_head_layer_reduces_to_attention_topk():
    """H = L = 1, rho = 1, lambda = 0: selection is plain top-K of the attention score."""
    for mode in (orc.SCORE_EQ1, orc.SCORE_CAUSAL_PROB):
        q, k, ns, nv, nt, gh, gw = _tiny_inputs(22, L=1, H=1, Hkv=1, grids=((8, 8),), NT=(6,))
        p = orc.Params(score_mode=mode, flags=orc.NO_RELIABILITY | orc.NO_NOVELTY)
        out = orc.decide(q, k, ns, nv, nt, gh, gw, [13], H_kv=1, params=p)
        assert out["keep"][0].tolist() == orc.topk(out["a"][0, 0], 13).tolist()


def test_compaction_rows_brute_force():
    keeps = [np.array([1, 4]), np.array([0])]
    ns, nv, nt = [2, 1], [5, 3], [2, 1]
    src = np.arange(sum(a + b + c for a, b, c in zip(ns, nv, nt)))[:, None] * 10
    got = orc.compact(src, ns, nv, nt, keeps)[:, 0].tolist()
    want = []
    off = 0
    for b in range(2):
        for j in range(ns[b] + nv[b] + nt[b]):
            if j < ns[b] or j >= ns[b] + nv[b] or (j - ns[b]) in keeps[b].tolist():
                want.append((off + j) * 10)
        off += ns[b] + nv[b] + nt[b]
    assert got == want
    assert orc.position_ids(ns, nv, nt, keeps).tolist() == [0, 1, 3, 6, 7, 8, 0, 1, 4]


def test_ds_generic_three_element_frame_example():
    """The generic rule handles composite focal sets (Eq. 5 style masses)."""
    A, B, C = "a", "b", "c"
    m1 = {frozenset({A, B}): 0.4, frozenset({C}): 0.6}
    m2 = {frozenset({A}): 0.5, frozenset({A, B, C}): 0.5}
    K = ds.conflict(m1, m2)
    assert K == pytest.approx(0.3)
    m = ds.combine(m1, m2)
    assert m[frozenset({A})] == pytest.approx(0.2 / 0.7)
    assert m[frozenset({A, B})] == pytest.approx(0.2 / 0.7)
    assert m[frozenset({C})] == pytest.approx(0.3 / 0.7)
    assert ds.belief(m, frozenset({A, B})) == pytest.approx(0.4 / 0.7)
    assert ds.plausibility(m, frozenset({B})) == pytest.approx(0.2 / 0.7)


def test_causal_row_lse_matches_library_logsumexp():
    """Sec. 3.1: each text row's normaliser over its causal prefix, against
    scipy's logsumexp of the visible logits taken row by row."""
    from scipy.special import logsumexp
    r = np.random.default_rng(11)
    Q = r.normal(size=(5, 16))
    K = r.normal(size=(12, 16))
    lse = orc.causal_row_lse(Q, K, 6)
    for t in range(5):
        vis = [float(Q[t] @ K[j]) / 4.0 for j in range(6 + t + 1)]
        assert abs(lse[t] - logsumexp(vis)) < 1e-12


def test_causal_row_lse_reconstructs_attention_rows():
    """exp(logit - lse) over the visible prefix is the causal softmax row, and
    a row that sees a single key has lse equal to that key's logit."""
    r = np.random.default_rng(12)
    Q = r.normal(size=(4, 8))
    K = r.normal(size=(9, 8))
    lse = orc.causal_row_lse(Q, K, 5)
    P = orc.causal_attention_rows(Q, K, 5)
    logits = Q @ K.T / np.sqrt(8)
    for t in range(4):
        n = 5 + t + 1
        assert np.allclose(np.exp(logits[t, :n] - lse[t]), P[t, :n], atol=1e-14)
        assert np.all(P[t, n:] == 0)
    one = orc.causal_row_lse(Q[:1], K, 0)
    assert abs(one[0] - logits[0, 0]) < 1e-14


# ------------------------------------------------------ the layer's attention
def test_attention_output_with_identity_values_is_the_softmax_rows():
    """V = identity: O = P, each row a textbook softmax of the visible logits
    (scipy), zero beyond the row's own position; lse is scipy's logsumexp."""
    from scipy.special import logsumexp
    r = _rng(40)
    T, d = 9, 8
    Q, K = r.normal(size=(T, d)), r.normal(size=(T, d))
    O, lse = orc.causal_attention_output(Q, K, np.eye(T))
    logits = Q @ K.T / math.sqrt(d)
    for p in range(T):
        np.testing.assert_allclose(O[p, :p + 1], sp_softmax(logits[p, :p + 1]), atol=1e-14)
        assert np.all(O[p, p + 1:] == 0)
        assert abs(lse[p] - logsumexp(logits[p, :p + 1])) < 1e-12


def test_attention_output_special_cases():
    r = _rng(41)
    T, d = 7, 4
    Q, K, V = r.normal(size=(T, d)), r.normal(size=(T, d)), r.normal(size=(T, 5))
    O, _ = orc.causal_attention_output(Q, K, V)
    np.testing.assert_allclose(O[0], V[0], atol=1e-15)             # the first row sees one key
    O2, _ = orc.causal_attention_output(Q, K, np.tile(V[3], (T, 1)))
    np.testing.assert_allclose(O2, np.tile(V[3], (T, 1)), atol=1e-14)   # equal values: O = v
    # brute force with math.exp for the last row
    lg = [sum(Q[T - 1, i] * K[j, i] for i in range(d)) / math.sqrt(d) for j in range(T)]
    w = [math.exp(x - max(lg)) for x in lg]
    want = [sum(w[j] * V[j, c] for j in range(T)) / sum(w) for c in range(5)]
    np.testing.assert_allclose(O[T - 1], want, atol=1e-13)


def test_attention_text_rows_give_the_score_and_row_lse():
    """The text rows of the layer's attention carry the decision's inputs:
    their lse equals causal_row_lse, and the mean of their probabilities on
    the visual keys (recovered as O with identity values) is a."""
    r = _rng(42)
    S, NV, NT, d = 3, 6, 4, 8
    T = S + NV + NT
    Q, K = r.normal(size=(T, d)), r.normal(size=(T, d))
    O, lse = orc.causal_attention_output(Q, K, np.eye(T))
    np.testing.assert_allclose(lse[S + NV:], orc.causal_row_lse(Q[S + NV:], K, S + NV), atol=1e-12)
    np.testing.assert_allclose(O[S + NV:, S:S + NV].mean(axis=0),
                               orc.score_causal_prob(Q[S + NV:], K, S, NV), atol=1e-15)
