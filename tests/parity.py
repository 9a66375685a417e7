"""Parity checks of the CUDA path against the CPU oracle.

Tolerances (floating point): every float output -- a, masses, p_bar, fused
masses, conflict K, q and q~ -- within max abs 1e-3 of the float64 oracle
(bf16 inputs, fp32 accumulation on the GPU).  Causal-probability scores are
also held to an elementwise relative bound, A_REL: a token's a is about
1/N_V (1.7e-3 on a 24 x 24 grid), the same size as the absolute tolerance, so
that tolerance alone cannot see a wrong score.  Dropping one text row from the
mean moves a by up to 2-3 % of its value on the LLaVA shapes, and a causal
mask one key short by 0.16 % (tests/test_parity_bounds.py); the GPU's own
error is about 1e-5 relative (fp32 sums of ex2.approx terms, relative error
~2^-22 each).

Discrete outputs, where floating point decides an integer:
  * cell representative b (Eqs. 20-21): where the oracle's best q in a cell
    leads the runner-up by more than TOL, the GPU must pick the same token;
    otherwise it must pick one of the tokens within TOL of the cell maximum.
  * retained set (Eq. 23): with the GPU's (validated) representatives, the
    oracle's q~ is formed in float64; thr is the midpoint of its K-th and
    (K+1)-th largest values.  Every token above thr + TOL must be kept and
    every token below thr - TOL dropped, so the sets are identical whenever
    the margin exceeds TOL; the set has exactly min(K, N_V) ascending entries.
  * compaction: bit-exact.
"""
from __future__ import annotations

import numpy as np

from oracle import e2s_oracle as orc

TOL = 1e-3
A_REL = 5e-4


def max_err(got, want) -> float:
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    assert got.shape == want.shape, (got.shape, want.shape)
    if got.size == 0:
        return 0.0
    assert np.all(np.isfinite(got)), "non-finite GPU output"
    return float(np.abs(got - want).max())


def assert_close(name, got, want, tol=TOL):
    e = max_err(got, want)
    if e > tol:
        g = np.asarray(got, dtype=np.float64)
        w = np.asarray(want, dtype=np.float64)
        d = np.abs(g - w)
        at = np.unravel_index(int(np.argmax(d)), d.shape)
        n_bad = int((d > tol).sum())
        raise AssertionError(f"{name}: max abs err {e:.3g} > {tol} at {tuple(int(i) for i in at)} "
                             f"(got {g[at]:.6g}, want {w[at]:.6g}; {n_bad} of {d.size} beyond)")
    return e


def check_a(got, want, causal: bool, tol=TOL, rel=A_REL):
    """a within the absolute tolerance, and for causal-probability scores
    (strictly positive) within `rel` of each oracle value."""
    e = assert_close("a", got, want, tol)
    if causal and np.size(want):
        g = np.asarray(got, dtype=np.float64)
        w = np.asarray(want, dtype=np.float64)
        assert np.all(w > 0), "causal-probability scores must be positive"
        r = float((np.abs(g - w) / w).max())
        assert r <= rel, f"a: max relative err {r:.3g} > {rel}"
    return e


def check_floats(gpu: dict, ref: dict, tol=TOL, mass=True):
    causal = ref.get("score_mode", orc.SCORE_CAUSAL_PROB) == orc.SCORE_CAUSAL_PROB
    errs = {"a": check_a(gpu["a"], ref["a"], causal, tol)}
    if mass and gpu.get("mass") is not None:
        m = gpu["mass"]
        errs["mass"] = assert_close("mass", m[..., :3], ref["mass"], tol)
        errs["p_bar"] = assert_close("p_bar", m[..., 3], ref["p_bar"], tol)
    errs["fused"] = assert_close("fused", gpu["fused"][:, :3], ref["fused"], tol)
    errs["K"] = assert_close("K", gpu["fused"][:, 3], ref["K"], tol)
    errs["q"] = assert_close("q", gpu["q"], ref["q"], tol)
    return errs


def check_selection(gpu_keep, gpu_q_tilde, ref_q, n_vis, grid_h, grid_w, keep, lam, G,
                    cand=None, tol=TOL):
    """Cell representatives, q~ and the retained set of every image."""
    off = 0
    for b in range(len(n_vis)):
        nv = int(n_vis[b])
        q = np.asarray(ref_q[off:off + nv], dtype=np.float64)
        raster = np.arange(nv) if cand is None else np.asarray(cand[b])
        cells = orc.cell_of(raster, int(grid_h[b]), int(grid_w[b]), G)
        qt_gpu = np.asarray(gpu_q_tilde[off:off + nv], dtype=np.float64)
        # representatives as chosen by the GPU: q~ - (1 - lam) q ~ lam
        b_gpu = (qt_gpu - (1 - lam) * q) > lam / 2 if lam > 0 else np.zeros(nv, bool)
        bind = np.zeros(nv)
        if lam > 0:
            for g in np.unique(cells):
                mem = np.nonzero(cells == g)[0]
                chosen = mem[b_gpu[mem]]
                assert chosen.size == 1, f"image {b} cell {g}: {chosen.size} representatives"
                qm = q[mem]
                best = qm.max()
                ok = mem[qm >= best - tol]
                assert chosen[0] in ok, f"image {b} cell {g}: rep {chosen[0]} not near-max"
                if ok.size == 1:
                    assert chosen[0] == ok[0]
                bind[chosen[0]] = 1.0
        qt = (1 - lam) * q + lam * bind
        assert_close(f"q_tilde[{b}]", qt_gpu, qt, tol)
        K = int(keep[b])
        kc = min(K, nv)
        kept = np.asarray(gpu_keep[b])
        assert kept.size == K
        assert np.all(kept[kc:] == -1)
        kept = kept[:kc]
        assert np.all(np.diff(kept) > 0), "keep_idx not strictly ascending"
        assert kept.size == 0 or (kept[0] >= 0 and kept[-1] < nv)
        if 0 < kc < nv:
            s = np.sort(qt)[::-1]
            thr = 0.5 * (s[kc - 1] + s[kc])
            mask = np.zeros(nv, bool)
            mask[kept] = True
            must = qt > thr + tol
            never = qt < thr - tol
            assert np.all(mask[must]), f"image {b}: a clearly retained token was dropped"
            assert not np.any(mask[never]), f"image {b}: a clearly pruned token was kept"
        off += nv


def clear_margin_images(ref, n_vis, keep, tol=TOL):
    """Images whose oracle K-th / (K+1)-th q~ margin exceeds tol."""
    out, off = [], 0
    for b in range(len(n_vis)):
        nv = int(n_vis[b])
        kc = min(int(keep[b]), nv)
        if 0 < kc < nv:
            s = np.sort(ref["q_tilde"][off:off + nv])[::-1]
            if s[kc - 1] - s[kc] > tol:
                out.append(b)
        else:
            out.append(b)
        off += nv
    return out


def oracle_keep_ok(ref, n_vis, keep, tol=TOL):
    """Whether the oracle's own K-th / (K+1)-th margin exceeds tol for every image."""
    return len(clear_margin_images(ref, n_vis, keep, tol)) == len(n_vis)


def check_topk_of_own_scores(gpu_keep, gpu_q_tilde, n_vis, keep):
    """The integer step taken in the kernel's precision: each image's retained
    set is the Top-K of the q~ the GPU wrote (float32, ties to the lower
    index), in ascending order."""
    off = 0
    for b in range(len(n_vis)):
        nv = int(n_vis[b])
        kc = min(int(keep[b]), nv)
        qt = np.asarray(gpu_q_tilde[off:off + nv], dtype=np.float32)
        order = np.lexsort((np.arange(nv), -qt.astype(np.float64)))
        want = np.sort(order[:kc])
        assert np.array_equal(np.asarray(gpu_keep[b])[:kc], want), f"image {b}: not Top-K of q~"
        off += nv
