"""Pins of the oracle's branches that the GPU parity tests lean on (CPU only).

Each pin compares a branch of the oracle with something other than its own
formula -- the definition of grouped-query attention, the generic Dempster
rule, a one-layer input, a pure-Python loop, a brute-force scan of the 2-D
grid -- and each has a planted mistake beside it that the pin must reject:

  * GQA head mapping (Sec. 3.1 with grouped KV heads): query head h reads kv
    head floor(h / group).  Pin: a GQA input equals the same input with every
    kv head repeated `group` times and run as multi-head attention.
  * Table 2, A4 (NO_CONFLICT): q is the plausibility Pl of Eq. 18 of the fused
    mass, with no conflict term.  Pin: Pl from the generic rule (Eqs. 3-4, 7)
    enumerated over focal sets, layer by layer.
  * Table 2, A3 (NO_LAYER_FUSION): only the current (last) evidence layer; a
    carried prior is ignored.  Pin: the decision on a one-layer input holding
    only that layer, without prior.
  * Table 2, A1 (VANILLA): q is the mean of a over layers and heads and the
    novelty bonus is off.  Pin: a pure-Python triple loop and a greedy Top-K,
    with a large lambda that must have no effect.
  * Progressive candidates (Algorithm 1, V <- TopK; Sec. 4.3): the spatial
    cells of a surviving token come from its ORIGINAL raster position.  Pin:
    a brute-force scan of the h x w grid in G x G blocks.
"""
import numpy as np
import pytest

from oracle import ds_generic as ds
from oracle import e2s_oracle as orc

I_, U_ = "I", "U"
THETA = frozenset({I_, U_})


def _bits(x):
    return (np.asarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def _inputs(seed, *, L=2, H=6, H_kv=2, grids=((8, 12),), NT=(5,), S=3, d=16, spike=True):
    """Tiny packed batch.  With `spike`, a few visual keys per kv head are
    pushed along a shared direction that the queries also carry, so the
    attention is peaked and the evidence is not uniform."""
    r = np.random.default_rng(seed)
    n_vis = [h * w for h, w in grids]
    T = [S + nv + nt for nv, nt in zip(n_vis, NT)]
    q = r.normal(size=(L, sum(NT), H, d)) * 0.5
    k = r.normal(size=(L, sum(T), H_kv, d)) * 0.5
    if spike:
        off = 0
        for b, nv in enumerate(n_vis):
            for l in range(L):
                for g in range(H_kv):
                    u = r.normal(size=d)
                    u /= np.linalg.norm(u)
                    hot = r.choice(nv, size=max(1, nv // 8), replace=False)
                    k[l, off + S + hot, g] += 3.0 * u
            off += T[b]
        x0 = 0
        for b in range(len(n_vis)):
            q[:, x0:x0 + NT[b]] += r.uniform(0, 2, size=(L, 1, H, 1)) * r.normal(size=(1, 1, H, d))
            x0 += NT[b]
    return (_bits(q), _bits(k), [S] * len(grids), n_vis, list(NT),
            [g[0] for g in grids], [g[1] for g in grids])


# ------------------------------------------------------------------ GQA mapping
def _gqa_pin(decide_fn, mode):
    """a, q and the keep set of a GQA input equal those of the MHA input whose
    kv head h is kv head floor(h / group) of the GQA input."""
    H, H_kv = 6, 2
    group = H // H_kv
    q, k, ns, nv, nt, gh, gw = _inputs(30, H=H, H_kv=H_kv, grids=((8, 12), (4, 4)), NT=(5, 3))
    k_mha = np.repeat(k, group, axis=2)            # k_mha[..., h, :] = k[..., h // group, :]
    p = orc.Params(score_mode=mode)
    g = decide_fn(q, k, ns, nv, nt, gh, gw, [20, 5], H_kv=H_kv, params=p)
    m = decide_fn(q, k_mha, ns, nv, nt, gh, gw, [20, 5], H_kv=H, params=p)
    np.testing.assert_allclose(g["a"], m["a"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(g["q"], m["q"], rtol=0, atol=1e-14)
    for x, y in zip(g["keep"], m["keep"]):
        assert x.tolist() == y.tolist()


@pytest.mark.parametrize("mode", [orc.SCORE_EQ1, orc.SCORE_CAUSAL_PROB])
def test_gqa_equals_mha_with_repeated_kv_heads(mode):
    _gqa_pin(orc.decide, mode)


def test_gqa_row_lse_equals_mha_with_repeated_kv_heads():
    q, k, ns, nv, nt, _, _ = _inputs(31, H=6, H_kv=3)
    lse_g = orc.text_row_lse(q, k, ns, nv, nt, H_kv=3)
    lse_m = orc.text_row_lse(q, np.repeat(k, 2, axis=2), ns, nv, nt, H_kv=6)
    np.testing.assert_allclose(lse_g, lse_m, rtol=0, atol=1e-14)


def test_gqa_modulo_head_mapping_is_caught(monkeypatch):
    """Query head h reading kv head h % H_kv (interleaved groups) fails the pin."""
    def bad_image_scores(q_text, k, b, lay, H_kv, score_mode):
        L, _, H, d = q_text.shape
        S, N_V, N_T = int(lay["n_sys"][b]), int(lay["n_vis"][b]), int(lay["n_text"][b])
        t0, x0 = int(lay["tok_off"][b]), int(lay["text_off"][b])
        a = np.zeros((L, H, N_V))
        for l in range(L):
            for h in range(H):
                Q = orc.widen_bf16(q_text[l, x0:x0 + N_T, h])
                Kh = orc.widen_bf16(k[l, t0:t0 + S + N_V + N_T, h % H_kv])
                a[l, h] = orc.score_causal_prob(Q, Kh, S, N_V)
        return a
    _gqa_pin(orc.decide, orc.SCORE_CAUSAL_PROB)
    monkeypatch.setattr(orc, "image_scores", bad_image_scores)
    with pytest.raises(AssertionError):
        _gqa_pin(orc.decide, orc.SCORE_CAUSAL_PROB)


# ------------------------------------------------------------------ A4: NO_CONFLICT
def _generic(m):
    return {frozenset({I_}): float(m[0]), frozenset({U_}): float(m[1]), THETA: float(m[2])}


def _generic_pl(masses):
    """Pl(I) of the layer masses [L][3] fused in order by the generic rule."""
    acc = _generic(masses[0])
    for l in range(1, len(masses)):
        acc = ds.combine(acc, _generic(masses[l]))
    return ds.plausibility(acc, frozenset({I_}))


def _check_no_conflict(out):
    for n in range(out["q"].size):
        assert abs(out["q"][n] - _generic_pl(out["mass"][:, n])) < 1e-12, n


def test_no_conflict_priority_is_generic_plausibility():
    q, k, ns, nv, nt, gh, gw = _inputs(32, L=3)
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [17], H_kv=2,
                     params=orc.Params(flags=orc.NO_CONFLICT))
    _check_no_conflict(out)
    full = orc.decide(q, k, ns, nv, nt, gh, gw, [17], H_kv=2, params=orc.Params())
    assert np.abs(full["q"] - out["q"]).max() > 1e-3       # the flag changes q


def test_no_conflict_mistakes_are_caught():
    q, k, ns, nv, nt, gh, gw = _inputs(32, L=3)
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [17], H_kv=2,
                     params=orc.Params(flags=orc.NO_CONFLICT))
    for bad_q in (orc.priority(out["pl"], out["K"]),          # flag ignored: Eq. 19 kept
                  out["bel"]):                                  # Bel (Eq. 17) instead of Pl
        bad = dict(out, q=bad_q)
        with pytest.raises(AssertionError):
            _check_no_conflict(bad)


# ------------------------------------------------------------------ A3: NO_LAYER_FUSION
def _check_same_decision(x, y):
    for key in ("fused", "K", "q", "q_tilde"):
        np.testing.assert_allclose(x[key], y[key], rtol=0, atol=1e-14, err_msg=key)
    for a, b in zip(x["keep"], y["keep"]):
        assert a.tolist() == b.tolist()


def _nlf_case():
    q, k, ns, nv, nt, gh, gw = _inputs(33, L=3)
    r = np.random.default_rng(5)
    prior = r.dirichlet([1.0, 1.0, 1.0], size=sum(nv))
    return q, k, ns, nv, nt, gh, gw, prior


def test_no_layer_fusion_equals_last_layer_alone():
    q, k, ns, nv, nt, gh, gw, prior = _nlf_case()
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [23], H_kv=2,
                     params=orc.Params(flags=orc.NO_LAYER_FUSION), prior=prior)
    last = orc.decide(q[-1:], k[-1:], ns, nv, nt, gh, gw, [23], H_kv=2, params=orc.Params())
    _check_same_decision(out, last)
    np.testing.assert_allclose(out["K"], 0.0)                # no combination happened


def test_no_layer_fusion_mistakes_are_caught():
    q, k, ns, nv, nt, gh, gw, prior = _nlf_case()
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [23], H_kv=2,
                     params=orc.Params(flags=orc.NO_LAYER_FUSION), prior=prior)
    first = orc.decide(q[:1], k[:1], ns, nv, nt, gh, gw, [23], H_kv=2, params=orc.Params())
    with_prior = orc.decide(q[-1:], k[-1:], ns, nv, nt, gh, gw, [23], H_kv=2,
                            params=orc.Params(), prior=prior)
    for bad in (first, with_prior):                          # wrong layer / prior fused in
        with pytest.raises(AssertionError):
            _check_same_decision(out, bad)


# ------------------------------------------------------------------ A1: VANILLA
def _check_vanilla(out, keep):
    a = out["a"]
    L, H, N = a.shape
    for n in range(N):
        s = 0.0
        for l in range(L):
            for h in range(H):
                s += a[l][h][n]
        assert abs(out["q"][n] - s / (L * H)) < 1e-12, n
    left, chosen = list(range(N)), []
    for _ in range(min(keep, N)):
        best = left[0]
        for n in left:
            if out["q"][n] > out["q"][best]:
                best = n
        chosen.append(best)
        left.remove(best)
    assert out["keep"][0].tolist() == sorted(chosen)


def test_vanilla_ranks_by_mean_attention_without_novelty():
    q, k, ns, nv, nt, gh, gw = _inputs(34, L=3)
    for mode in (orc.SCORE_EQ1, orc.SCORE_CAUSAL_PROB):
        out = orc.decide(q, k, ns, nv, nt, gh, gw, [19], H_kv=2,
                         params=orc.Params(lam=0.5, score_mode=mode, flags=orc.VANILLA))
        _check_vanilla(out, 19)
        np.testing.assert_allclose(out["q_tilde"], out["q"], rtol=0, atol=0)


def test_vanilla_mistakes_are_caught():
    q, k, ns, nv, nt, gh, gw = _inputs(34, L=3)
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [19], H_kv=2,
                     params=orc.Params(lam=0.5, flags=orc.VANILLA))
    a = out["a"]
    # mean over heads of the last layer only
    bad = dict(out, q=a[-1].mean(axis=0))
    with pytest.raises(AssertionError):
        _check_vanilla(bad, 19)
    # the novelty bonus left on: the keep set follows q~ with representatives
    cells = orc.cell_of(np.arange(a.shape[2]), gh[0], gw[0], 4)
    qt = orc.adjusted_priority(out["q"], orc.representative_indicator(out["q"], cells), 0.5)
    bad = dict(out, keep=[orc.topk(qt, 19)])
    with pytest.raises(AssertionError):
        _check_vanilla(bad, 19)


# ------------------------------------------------------------------ progressive candidates
def _grid_representatives(q, cand, h, w, bh, bw):
    """Brute force over the 2-D grid: place each surviving slot at its original
    (row, col); the cells are the bh x bw blocks of a grid that G divides; the
    representative is the highest q in the block (lowest slot on ties)."""
    where = {int(c): s for s, c in enumerate(cand)}
    b = np.zeros(len(cand))
    for r0 in range(0, h, bh):
        for c0 in range(0, w, bw):
            best = None
            for i in range(r0, r0 + bh):
                for j in range(c0, c0 + bw):
                    s = where.get(i * w + j)
                    if s is None:
                        continue
                    if best is None or q[s] > q[best] or (q[s] == q[best] and s < best):
                        best = s
            if best is not None:
                b[best] = 1.0
    return b


def _cand_case(seed=35, G=4, h=8, w=12, keep=9):
    """One image on an h x w grid; a random ascending subset of its visual
    tokens survived an earlier step.  The reduced sequence holds only their
    keys, in raster order, between the system and text keys."""
    q, k, ns, nv, nt, _, _ = _inputs(seed, L=2, grids=((h, w),))
    r = np.random.default_rng(seed)
    cand = np.sort(r.choice(h * w, size=(h * w) // 2 + 3, replace=False))
    S = ns[0]
    rows = np.concatenate([np.arange(S), S + cand, S + h * w + np.arange(nt[0])])
    k_red = k[:, rows]
    return q, k_red, ns, [cand.size], nt, [h], [w], cand, keep


def _check_cand(out, cand, h, w, G, keep, lam=0.1):
    b = _grid_representatives(out["q"], cand, h, w, h // G, w // G)
    assert out["b"].tolist() == b.tolist()
    qt = (1 - lam) * out["q"] + lam * b
    left, chosen = list(range(len(cand))), []
    for _ in range(min(keep, len(cand))):
        best = left[0]
        for n in left:
            if qt[n] > qt[best]:
                best = n
        chosen.append(best)
        left.remove(best)
    assert out["keep"][0].tolist() == sorted(chosen)


def test_candidates_use_cells_of_original_raster():
    q, k, ns, nv, nt, gh, gw, cand, keep = _cand_case()
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [keep], H_kv=2, params=orc.Params(), cand=[cand])
    _check_cand(out, cand, gh[0], gw[0], 4, keep)


def test_candidates_slot_index_cells_are_caught(monkeypatch):
    """Cells taken from the slot index instead of the original raster index."""
    q, k, ns, nv, nt, gh, gw, cand, keep = _cand_case()
    real = orc.cell_of
    monkeypatch.setattr(orc, "cell_of", lambda raster, h, w, G: real(np.arange(len(raster)), h, w, G))
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [keep], H_kv=2, params=orc.Params(), cand=[cand])
    with pytest.raises(AssertionError):
        _check_cand(out, cand, gh[0], gw[0], 4, keep)


def test_candidates_transposed_grid_is_caught(monkeypatch):
    """Cells from a grid read as w x h (rows and columns swapped)."""
    q, k, ns, nv, nt, gh, gw, cand, keep = _cand_case()
    real = orc.cell_of
    monkeypatch.setattr(orc, "cell_of", lambda raster, h, w, G: real(raster, w, h, G))
    out = orc.decide(q, k, ns, nv, nt, gh, gw, [keep], H_kv=2, params=orc.Params(), cand=[cand])
    with pytest.raises(AssertionError):
        _check_cand(out, cand, gh[0], gw[0], 4, keep)
