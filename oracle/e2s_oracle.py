"""Float64 CPU oracle of the E2S-Pruner pruning decision (test infrastructure).

Follows the paper step by step, in the order of Algorithm 1:
  Sec. 3.1 Eq. 1            text-to-visual score a_{l,h,n}
  Sec. 4.1 Eqs. 8-11        normalise r, support p, reliability rho, layer mass m
  Sec. 4.2 Eqs. 12-19       Dempster-Shafer fusion across layers, Bel, Pl, priority q
  Sec. 4.3 Eqs. 20-23       spatial cell representative, indicator b, q~, Top-K
and the compaction of the retained rows that the shortened sequence implies
(Sec. 4 opening paragraph; Sec. 5.1.2 pruning settings).  causal_attention_output
and attention_layer give the pruning layer's own causal attention (output and
row normalisers), whose text rows the score reads.

Readings where the paper is silent or ambiguous (each one is listed in the
design notes as well):
  * score mode CAUSAL_PROB: softmax of Q_text K^T / sqrt(d) over each text
    row's full causal key prefix, keep the visual columns, mean over text rows.
    Text row t (0-based) sits at position S + N_V + t and sees keys 0..S+N_V+t.
    Mode EQ1 is Eq. 1 literally (mean of pre-softmax logits).
  * norm RENORM (default with CAUSAL_PROB): r = a / sum(a) over the
    candidates, instead of Eq. 8's softmax, which is degenerate on
    probabilities.  If sum(a) <= 0, r is uniform (1/N_l).
  * p-bar in Eqs. 10-11 is the arithmetic mean of p over the H query heads.
  * N_l in Eq. 9 is the number of candidate visual tokens of the image.
  * GQA: evidence is per query head h, using kv head floor(h / (H / H_kv)).
  * K^{(1)} = 0 for the first layer (no combination yet), so q = Pl.
  * Total conflict (1 - K <= 0): fused mass becomes vacuous (0, 0, 1), K = 1.
  * q uses the conflict K of the latest combination only.
  * Cell of grid point (i, j) on an h x w grid: (floor(i G / h), floor(j G / w)).
  * Ties (cell argmax and Top-K) go to the lower index; Top-K returns its
    indices in ascending order.
  * Ablations (Table 2): NO_RELIABILITY rho = 1; NO_LAYER_FUSION uses the
    last layer only; NO_CONFLICT q = Pl; NO_NOVELTY lambda = 0; VANILLA ranks
    by mean over layers and heads of a, with lambda = 0.  NO_LAYER_FUSION
    also ignores a carried prior (only the current layer's evidence).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional

import numpy as np

SCORE_EQ1 = "eq1"
SCORE_CAUSAL_PROB = "causal_prob"
NORM_SOFTMAX = "softmax"
NORM_RENORM = "renorm"

NO_RELIABILITY = 1
NO_LAYER_FUSION = 2
NO_CONFLICT = 4
NO_NOVELTY = 8
VANILLA = 16


def widen_bf16(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64, exactly."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------
# Sec. 3.1, Eq. 1 -- text-to-visual score
# --------------------------------------------------------------------------
def score_eq1(Q: np.ndarray, K_vis: np.ndarray) -> np.ndarray:
    """Eq. 1: a_n = (1/N_T) sum_t Q_t K_{v_n}^T / sqrt(d).

    Q: [N_T, d] text queries of one head; K_vis: [N_V, d] visual keys.
    """
    d = Q.shape[1]
    logits = Q @ K_vis.T / np.sqrt(d)          # [N_T, N_V]
    return logits.mean(axis=0)


def causal_attention_rows(Q: np.ndarray, K_all: np.ndarray, first_text_pos: int) -> np.ndarray:
    """Attention probabilities of the text rows over their causal prefixes.

    Row t is the text token at position first_text_pos + t; it attends to
    keys 0..first_text_pos + t.  Returns P [N_T, T] (zeros where masked).
    """
    d = Q.shape[1]
    T = K_all.shape[0]
    logits = Q @ K_all.T / np.sqrt(d)          # [N_T, T]
    pos = first_text_pos + np.arange(Q.shape[0])
    visible = np.arange(T)[None, :] <= pos[:, None]
    z = np.where(visible, logits, -np.inf)
    z = z - z.max(axis=1, keepdims=True)
    e = np.where(visible, np.exp(z), 0.0)
    return e / e.sum(axis=1, keepdims=True)


def causal_row_lse(Q: np.ndarray, K_all: np.ndarray, first_text_pos: int) -> np.ndarray:
    """Natural-log normaliser of each text row's causal softmax (Sec. 3.1):
    lse_t = log sum_{j <= first_text_pos + t} exp(Q_t K_j / sqrt(d)), so that
    P_{t,j} = exp(Q_t K_j / sqrt(d) - lse_t).  A flash-attention forward of the
    layer returns this value for every query row; the score can start from it.
    """
    d = Q.shape[1]
    T = K_all.shape[0]
    logits = Q @ K_all.T / np.sqrt(d)          # [N_T, T]
    pos = first_text_pos + np.arange(Q.shape[0])
    visible = np.arange(T)[None, :] <= pos[:, None]
    z = np.where(visible, logits, -np.inf)
    m = z.max(axis=1)
    return m + np.log(np.exp(z - m[:, None]).sum(axis=1))


def causal_attention_output(Q_all: np.ndarray, K_all: np.ndarray, V_all: np.ndarray):
    """Causal self-attention of one head over one image (Sec. 3.1): row p
    attends to keys 0..p with weights softmax_j(Q_p K_j / sqrt(d)); returns
    (O [T, d] = P V, lse [T] natural-log normaliser of each row)."""
    d = Q_all.shape[1]
    T = K_all.shape[0]
    logits = Q_all @ K_all.T / np.sqrt(d)      # [T, T]
    visible = np.arange(T)[None, :] <= np.arange(Q_all.shape[0])[:, None]
    z = np.where(visible, logits, -np.inf)
    m = z.max(axis=1)
    e = np.where(visible, np.exp(z - m[:, None]), 0.0)
    s = e.sum(axis=1)
    return (e / s[:, None]) @ V_all, m + np.log(s)


def score_causal_prob(Q: np.ndarray, K_all: np.ndarray, S: int, N_V: int) -> np.ndarray:
    """a_n = (1/N_T) sum_t P_{t, S+n}: mean text-to-visual attention probability."""
    P = causal_attention_rows(Q, K_all, S + N_V)
    return P[:, S:S + N_V].mean(axis=0)


# --------------------------------------------------------------------------
# Sec. 4.1, Eqs. 8-11 -- per-layer evidence
# --------------------------------------------------------------------------
def normalise_softmax(a: np.ndarray) -> np.ndarray:
    """Eq. 8: r_n = exp(a_n) / sum_j exp(a_j) over the candidate tokens."""
    e = np.exp(a - a.max())
    return e / e.sum()


def normalise_renorm(a: np.ndarray) -> np.ndarray:
    """r_n = a_n / sum_j a_j (reading of Eq. 8 for probability scores)."""
    s = a.sum()
    if s <= 0.0:
        return np.full_like(a, 1.0 / a.size)
    return a / s


def support(r: np.ndarray, N_l: int) -> np.ndarray:
    """Eq. 9: p = N_l r / (1 + N_l r); r = 1/N_l gives p = 1/2."""
    return N_l * r / (1.0 + N_l * r)


def reliability(p: np.ndarray):
    """Eq. 10 for every token at once.

    p: [H, N] supports of the H heads.  Returns (rho [N], p_bar [N]) with
    rho = (2/H)|sum_h (p_h - 1/2)| * (1 - (2/H) sum_h |p_h - p_bar|).
    """
    H = p.shape[0]
    p_bar = p.mean(axis=0)
    clarity = (2.0 / H) * np.abs((p - 0.5).sum(axis=0))
    consistency = 1.0 - (2.0 / H) * np.abs(p - p_bar[None, :]).sum(axis=0)
    return clarity * consistency, p_bar


def layer_mass(rho: np.ndarray, p_bar: np.ndarray) -> np.ndarray:
    """Eq. 11: (m(I), m(U), m(Theta)) = (rho p_bar, rho (1 - p_bar), 1 - rho). Returns [N, 3]."""
    return np.stack([rho * p_bar, rho * (1.0 - p_bar), 1.0 - rho], axis=-1)


# --------------------------------------------------------------------------
# Sec. 4.2, Eqs. 12-19 -- layer-wise Dempster-Shafer fusion
# --------------------------------------------------------------------------
def conflict(prev: np.ndarray, m: np.ndarray) -> np.ndarray:
    """Eq. 13: K = m~(I) m(U) + m~(U) m(I)."""
    return prev[..., 0] * m[..., 1] + prev[..., 1] * m[..., 0]


def dempster_combine(prev: np.ndarray, m: np.ndarray):
    """Eqs. 13-16 on frame {I, U}: returns (fused [..., 3], K [...]).

    Total conflict (1 - K <= 0) yields the vacuous mass (0, 0, 1) and K = 1.
    """
    K = conflict(prev, m)
    one_minus_K = 1.0 - K
    I = prev[..., 0] * m[..., 0] + prev[..., 0] * m[..., 2] + prev[..., 2] * m[..., 0]   # Eq. 14
    U = prev[..., 1] * m[..., 1] + prev[..., 1] * m[..., 2] + prev[..., 2] * m[..., 1]   # Eq. 15
    Th = prev[..., 2] * m[..., 2]                                                        # Eq. 16
    total = one_minus_K <= 0.0
    safe = np.where(total, 1.0, one_minus_K)
    fused = np.stack([I / safe, U / safe, Th / safe], axis=-1)
    fused = np.where(total[..., None], np.array([0.0, 0.0, 1.0]), fused)
    K = np.where(total, 1.0, K)
    return fused, K


def fuse_layers(masses: np.ndarray, prior: Optional[np.ndarray] = None):
    """Eqs. 12-16 recursively over the evidence layers, in order.

    masses: [L, N, 3].  Without a prior, m~^{(1)} = m_1 (Eq. 12) and K^{(1)} = 0.
    With a prior (fused state carried from an earlier pruning step), every
    layer, the first included, is combined with the running state.
    Returns (fused [N, 3], K of the latest combination [N]).
    """
    if prior is None:
        fused = masses[0].copy()
        K = np.zeros(masses.shape[1])
        start = 1
    else:
        fused = prior.copy()
        K = np.zeros(masses.shape[1])
        start = 0
    for l in range(start, masses.shape[0]):
        fused, K = dempster_combine(fused, masses[l])
    return fused, K


def belief(fused: np.ndarray) -> np.ndarray:
    """Eq. 17: Bel(I) = m~(I)."""
    return fused[..., 0]


def plausibility(fused: np.ndarray) -> np.ndarray:
    """Eq. 18: Pl(I) = m~(I) + m~(Theta) = 1 - m~(U)."""
    return fused[..., 0] + fused[..., 2]


def priority(Pl: np.ndarray, K: np.ndarray) -> np.ndarray:
    """Eq. 19: q = 1 - (1 - Pl)(1 - K)."""
    return 1.0 - (1.0 - Pl) * (1.0 - K)


# --------------------------------------------------------------------------
# Sec. 4.3, Eqs. 20-23 -- spatial novelty and Top-K
# --------------------------------------------------------------------------
def cell_of(raster: np.ndarray, h: int, w: int, G: int) -> np.ndarray:
    """Cell id of grid point n = i*w + j in the G x G partition of an h x w grid."""
    i = raster // w
    j = raster % w
    return (i * G // h) * G + (j * G // w)


def representative_indicator(q: np.ndarray, cells: np.ndarray) -> np.ndarray:
    """Eqs. 20-21: b_n = 1 for the arg-max-q token of every occupied cell.

    Ties go to the lower candidate index.
    """
    b = np.zeros(q.size)
    for g in np.unique(cells):
        members = np.nonzero(cells == g)[0]          # ascending
        best = members[np.argmax(q[members])]        # first maximum -> lowest index
        b[best] = 1.0
    return b


def adjusted_priority(q: np.ndarray, b: np.ndarray, lam: float) -> np.ndarray:
    """Eq. 22: q~ = (1 - lambda) q + lambda b."""
    return (1.0 - lam) * q + lam * b


def topk(q_tilde: np.ndarray, K: int) -> np.ndarray:
    """Eq. 23: the K candidates of largest q~ (ties: lower index), ascending."""
    K = max(0, min(int(K), q_tilde.size))
    idx = np.arange(q_tilde.size)
    order = np.lexsort((idx, -q_tilde))
    return np.sort(order[:K])


# --------------------------------------------------------------------------
# Compaction of the retained rows
# --------------------------------------------------------------------------
def retained_rows(S: int, N_V: int, N_T: int, keep: np.ndarray) -> np.ndarray:
    """Image-local source rows of the shortened sequence, in order:
    [0, S) system, S + keep (ascending), [S + N_V, S + N_V + N_T) text."""
    return np.concatenate([np.arange(S), S + np.asarray(keep, dtype=np.int64),
                           S + N_V + np.arange(N_T)]).astype(np.int64)


# --------------------------------------------------------------------------
# The whole decision (Algorithm 1, one pruning step over L evidence layers)
# --------------------------------------------------------------------------
@dataclasses.dataclass
class Params:
    lam: float = 0.1
    G: int = 4
    score_mode: str = SCORE_CAUSAL_PROB
    norm_mode: Optional[str] = None      # None: RENORM for CAUSAL_PROB, SOFTMAX for EQ1
    flags: int = 0

    def norm(self) -> str:
        if self.norm_mode is not None:
            return self.norm_mode
        return NORM_RENORM if self.score_mode == SCORE_CAUSAL_PROB else NORM_SOFTMAX


def image_scores(q_text, k, b, lay, H_kv, score_mode) -> np.ndarray:
    """a [L, H, N_V] of image b (Eq. 1 or the causal-prefix reading)."""
    L, _, H, d = q_text.shape
    group = H // H_kv
    S, N_V, N_T = int(lay["n_sys"][b]), int(lay["n_vis"][b]), int(lay["n_text"][b])
    t0, x0 = int(lay["tok_off"][b]), int(lay["text_off"][b])
    T = S + N_V + N_T
    a = np.zeros((L, H, N_V))
    for l in range(L):
        for h in range(H):
            Q = widen_bf16(q_text[l, x0:x0 + N_T, h])
            if score_mode == SCORE_EQ1:
                a[l, h] = score_eq1(Q, widen_bf16(k[l, t0 + S:t0 + S + N_V, h // group]))
            else:
                a[l, h] = score_causal_prob(Q, widen_bf16(k[l, t0:t0 + T, h // group]), S, N_V)
    return a


def text_row_lse(q_text, k, n_sys, n_vis, n_text, *, H_kv: int) -> np.ndarray:
    """lse [L, H, sum N_T] of every text row of a packed batch (causal_row_lse
    per image, layer and query head), laid out as the rows of q_text."""
    L, sum_text, H, d = q_text.shape
    group = H // H_kv
    out = np.zeros((L, H, sum_text))
    t0 = x0 = 0
    for b in range(len(n_sys)):
        S, N_V, N_T = int(n_sys[b]), int(n_vis[b]), int(n_text[b])
        T = S + N_V + N_T
        for l in range(L):
            for h in range(H):
                Q = widen_bf16(q_text[l, x0:x0 + N_T, h])
                out[l, h, x0:x0 + N_T] = causal_row_lse(
                    Q, widen_bf16(k[l, t0:t0 + T, h // group]), S + N_V)
        t0 += T
        x0 += N_T
    return out


def attention_layer(q_all, k, v, n_sys, n_vis, n_text, *, H_kv: int):
    """Causal attention of every image, layer and query head of a packed batch:
    q_all uint16 [L, sum T, H, d], k / v uint16 [L, sum T, H_kv, d] (bf16 bits).
    Returns O [L, sum T, H, d] and lse [L, H, sum T] (float64); query head h
    reads kv head floor(h / (H / H_kv))."""
    L, sum_T, H, d = q_all.shape
    group = H // H_kv
    O = np.zeros((L, sum_T, H, d))
    lse = np.zeros((L, H, sum_T))
    t0 = 0
    for b in range(len(n_sys)):
        T = int(n_sys[b]) + int(n_vis[b]) + int(n_text[b])
        for l in range(L):
            for h in range(H):
                o, ls = causal_attention_output(widen_bf16(q_all[l, t0:t0 + T, h]),
                                                widen_bf16(k[l, t0:t0 + T, h // group]),
                                                widen_bf16(v[l, t0:t0 + T, h // group]))
                O[l, t0:t0 + T, h] = o
                lse[l, h, t0:t0 + T] = ls
        t0 += T
    return O, lse


def image_evidence(a: np.ndarray, params: Params) -> Dict[str, np.ndarray]:
    """Eqs. 8-11 for every layer of one image: a [L, H, N] -> r, p, rho, p_bar, m."""
    L, H, N = a.shape
    r = np.zeros_like(a)
    for l in range(L):
        for h in range(H):
            r[l, h] = normalise_softmax(a[l, h]) if params.norm() == NORM_SOFTMAX \
                else normalise_renorm(a[l, h])
    p = support(r, N)
    rho = np.zeros((L, N))
    p_bar = np.zeros((L, N))
    for l in range(L):
        rho[l], p_bar[l] = reliability(p[l])
    if params.flags & NO_RELIABILITY:
        rho[:] = 1.0
    m = np.stack([layer_mass(rho[l], p_bar[l]) for l in range(L)])
    return {"r": r, "p": p, "rho": rho, "p_bar": p_bar, "mass": m}


def decide(q_text, k, n_sys, n_vis, n_text, grid_h, grid_w, keep, *, H_kv: int,
           params: Params = Params(), cand: Optional[List[np.ndarray]] = None,
           prior: Optional[np.ndarray] = None) -> Dict[str, object]:
    """One pruning decision for a packed batch.

    q_text uint16 [L, sum N_T, H, d], k uint16 [L, sum T, H_kv, d] (bf16 bits).
    cand[b] (optional): original raster index of each visual slot of image b
    (a progressive step after earlier pruning); default 0..N_V-1.
    prior (optional): [sum N_V, 3] fused mass carried from the previous step.
    Returns packed per-token arrays and per-image keep lists.
    """
    n_sys, n_vis, n_text = (np.asarray(x, dtype=np.int64) for x in (n_sys, n_vis, n_text))
    T = n_sys + n_vis + n_text
    lay = {
        "n_sys": n_sys, "n_vis": n_vis, "n_text": n_text,
        "tok_off": np.concatenate([[0], np.cumsum(T)]),
        "vis_off": np.concatenate([[0], np.cumsum(n_vis)]),
        "text_off": np.concatenate([[0], np.cumsum(n_text)]),
    }
    L, _, H, _ = q_text.shape
    sum_vis = int(lay["vis_off"][-1])
    out = {k_: np.zeros(s) for k_, s in [
        ("a", (L, H, sum_vis)), ("p", (L, H, sum_vis)), ("rho", (L, sum_vis)),
        ("p_bar", (L, sum_vis)), ("mass", (L, sum_vis, 3)), ("fused", (sum_vis, 3)),
        ("K", (sum_vis,)), ("bel", (sum_vis,)), ("pl", (sum_vis,)), ("q", (sum_vis,)),
        ("b", (sum_vis,)), ("q_tilde", (sum_vis,))]}
    keeps = []
    lam = 0.0 if params.flags & (NO_NOVELTY | VANILLA) else params.lam
    for b in range(len(n_vis)):
        v0, v1 = int(lay["vis_off"][b]), int(lay["vis_off"][b + 1])
        a = image_scores(q_text, k, b, lay, H_kv, params.score_mode)
        ev = image_evidence(a, params)
        if params.flags & NO_LAYER_FUSION:
            fused, K = fuse_layers(ev["mass"][-1:], None)
        else:
            fused, K = fuse_layers(ev["mass"], None if prior is None else prior[v0:v1])
        Pl = plausibility(fused)
        q = Pl.copy() if params.flags & NO_CONFLICT else priority(Pl, K)
        if params.flags & VANILLA:
            q = a.mean(axis=(0, 1))
        raster = np.arange(v1 - v0) if cand is None else np.asarray(cand[b], dtype=np.int64)
        cells = cell_of(raster, int(grid_h[b]), int(grid_w[b]), params.G)
        bind = representative_indicator(q, cells)
        qt = adjusted_priority(q, bind, lam)
        keeps.append(topk(qt, int(keep[b])))
        out["a"][:, :, v0:v1] = a
        out["p"][:, :, v0:v1] = ev["p"]
        out["rho"][:, v0:v1] = ev["rho"]
        out["p_bar"][:, v0:v1] = ev["p_bar"]
        out["mass"][:, v0:v1] = ev["mass"]
        out["fused"][v0:v1] = fused
        out["K"][v0:v1] = K
        out["bel"][v0:v1] = belief(fused)
        out["pl"][v0:v1] = Pl
        out["q"][v0:v1] = q
        out["b"][v0:v1] = bind
        out["q_tilde"][v0:v1] = qt
    out["keep"] = keeps
    return out


def compact(src_rows: np.ndarray, n_sys, n_vis, n_text, keeps) -> np.ndarray:
    """Gather the retained rows of a packed [sum T, ...] tensor (any dtype)."""
    idx = []
    off = 0
    for b in range(len(n_vis)):
        S, N_V, N_T = int(n_sys[b]), int(n_vis[b]), int(n_text[b])
        idx.append(off + retained_rows(S, N_V, N_T, keeps[b]))
        off += S + N_V + N_T
    idx = np.concatenate(idx) if idx else np.zeros(0, dtype=np.int64)
    return src_rows[idx]


def position_ids(n_sys, n_vis, n_text, keeps) -> np.ndarray:
    """Image-local original positions of the retained rows, in output order."""
    return np.concatenate([retained_rows(int(n_sys[b]), int(n_vis[b]), int(n_text[b]), keeps[b])
                           for b in range(len(n_vis))]).astype(np.int64)
