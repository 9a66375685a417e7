"""Seeded synthetic inputs for the pruning decision.

This module only draws random numbers and lays them out; it contains none of
the pruning method's arithmetic.  Both the CUDA path (tests, bench) and the
CPU oracle consume what it produces, so it imports neither of them.

Recipe (stands in for the paper's VLM prefill on GQA/SQA/TextVQA/POPE/MME/
MMBench/AI2D images and prompts, which are not available; shapes follow the
LLaVA-1.5-7B and Qwen2-VL-7B settings of Sec. 4.1 and Table 5):

* Token layout per image: ``[system S][visual N_V on an h x w grid][text N_T]``
  (Sec. 3.1).  ``T = S + N_V + N_T`` keys; queries exist only for text rows.
* Queries and keys are i.i.d. normal with variance ``d**-0.5``
  (sigma = d**-0.25, so a random logit ``q.k/sqrt(d)`` has std ~0.09).
* One unit salience direction ``u`` per (image, layer, kv head).  Every salient
  visual key gets ``+4 * sigma * sqrt(d) * u``.  Every text query of query head
  h gets ``+g[l, h] * sigma * sqrt(d) * u`` with ``g ~ U[0, 1.5]`` per
  (layer, query head), so salient logits sit about ``4 g`` above background and
  heads differ in how clearly they see the planted tokens.
* Salient tokens are planted either at random grid positions or as blobs:
  the grid points nearest to random centres, split as evenly as possible.
* V rows and hidden states are N(0, 1); they are only copied.
* Every float is rounded to bf16 (round-to-nearest-even) and returned as its
  16-bit pattern in a ``uint16`` array.
* Generator: numpy PCG64 with seed ``1000 * config + image``; per-image shape
  draws (ragged N_T, dynamic-resolution grid) use the same seed's ``jumped()`` stream.
"""
from __future__ import annotations

import concurrent.futures as cf
import dataclasses
import os
from typing import List, Optional, Sequence

import numpy as np

D_HEAD = 128
SIGMA = D_HEAD ** -0.25


def bf16_bits(x: np.ndarray, chunk: int = 1 << 20) -> np.ndarray:
    """Round float32 values to bf16 (nearest-even) and return the bit patterns:
    (u + 0x7FFF + ((u >> 16) & 1)) >> 16 on the float's bits, in place over
    cache-sized chunks."""
    u = np.ascontiguousarray(x, dtype=np.float32).reshape(-1).view(np.uint32)
    out = np.empty(u.shape, dtype=np.uint16)
    tmp = np.empty(min(chunk, max(u.size, 1)), dtype=np.uint32)
    for s in range(0, u.size, chunk):
        e = min(s + chunk, u.size)
        r = tmp[:e - s]
        np.right_shift(u[s:e], 16, out=r)
        r &= np.uint32(1)
        r += np.uint32(0x7FFF)
        r += u[s:e]
        r >>= np.uint32(16)
        out[s:e] = r
    return out.reshape(np.shape(x))


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclasses.dataclass
class ImageSpec:
    n_sys: int
    grid_h: int
    grid_w: int
    n_text: int
    n_salient: int
    blobs: int           # 0 = random positions, else number of blobs
    keep: int            # K for this image

    @property
    def n_vis(self) -> int:
        return self.grid_h * self.grid_w

    @property
    def n_tok(self) -> int:
        return self.n_sys + self.n_vis + self.n_text


@dataclasses.dataclass
class Spec:
    name: str
    cfg_id: int
    L: int
    H: int
    H_kv: int
    hidden: int          # 0 = no hidden/V tensors (decision only)
    images: List[ImageSpec]
    d: int = D_HEAD

    @property
    def B(self) -> int:
        return len(self.images)


def round_half_even(x: float) -> int:
    return int(np.round(x))


def keep_for_ratio(n_vis: int, ratio: float) -> int:
    return round_half_even(ratio * n_vis)


def config_spec(cfg: int, *, batch: Optional[int] = None, keep: Optional[int] = None,
                images: Optional[int] = None, keep_ratio: Optional[float] = None,
                dynamic_grids: bool = False) -> Spec:
    """Specs for the five workload configurations.

    cfg 0: tiny decision, B=1, L=2, MHA 32x128, 35 + 24x24 + 32, 20 random salient, K=64.
    cfg 1: LLaVA-1.5-7B, B=1, L=3, D=4096, 35 + 24x24 + 64, 40 salient in 3 blobs, K in {192,128,64}.
    cfg 2: cfg 1 per image, B=32, N_T ~ U[16,128] ragged, K in {64,128}.
    cfg 3: Qwen2-VL-7B, B=16, D=3584, 28 q / 4 kv heads, L=3, grids from
           {16x16, 24x32, 32x32, 36x36}, N_T=64, K = round(64/576 * N_V).
           ``dynamic_grids`` draws any h, w in [12, 48] with h * w <= 1296 instead
           (merged-patch grids of arbitrary image sizes, mostly not divisible by
           G = 4); ``keep_ratio`` sets K = round(keep_ratio * N_V) (Sec. 4.5:
           reductions of 66.7 % and 77.8 % keep 1/3 and 2/9).
    cfg 4: MHA 32x128, L=4, B=8 alternating 48x48 / 64x64 grids, N_T=128,
           salient blobs covering 5% of the grid, K = round(0.11 * N_V).
    ``batch``/``images`` shrink the batch for oracle-sized parity runs.
    """
    if cfg == 0:
        k = 64 if keep is None else keep
        ims = [ImageSpec(35, 24, 24, 32, 20, 0, k)]
        return Spec("tiny", 0, 2, 32, 32, 0, ims)
    if cfg == 1:
        k = 64 if keep is None else keep
        ims = [ImageSpec(35, 24, 24, 64, 40, 3, k)]
        return Spec("llava-b1", 1, 3, 32, 32, 4096, ims)
    if cfg == 2:
        b = 32 if batch is None else batch
        k = 64 if keep is None else keep
        ims = []
        for i in range(b):
            r = np.random.Generator(np.random.PCG64(1000 * 2 + i).jumped())
            nt = int(r.integers(16, 129))
            ims.append(ImageSpec(35, 24, 24, nt, 40, 3, k))
        return Spec("llava-b32-ragged", 2, 3, 32, 32, 4096, ims)
    if cfg == 3:
        b = 16 if batch is None else batch
        grids = [(16, 16), (24, 32), (32, 32), (36, 36)]
        ratio = 64 / 576 if keep_ratio is None else keep_ratio
        ims = []
        for i in range(b):
            r = np.random.Generator(np.random.PCG64(1000 * 3 + i).jumped())
            if dynamic_grids:
                while True:
                    gh, gw = int(r.integers(12, 49)), int(r.integers(12, 49))
                    if gh * gw <= 1296:
                        break
            else:
                gh, gw = grids[int(r.integers(0, 4))]
            nv = gh * gw
            ims.append(ImageSpec(35, gh, gw, 64, round_half_even(40 * nv / 576), 3,
                                 keep_for_ratio(nv, ratio) if keep is None else keep))
        name = "qwen2vl-gqa-dynres" if dynamic_grids else "qwen2vl-gqa-ragged"
        return Spec(name, 3, 3, 28, 4, 3584, ims)
    if cfg == 4:
        b = 8 if batch is None else batch
        ims = []
        for i in range(b):
            g = 48 if i % 2 == 0 else 64
            nv = g * g
            ims.append(ImageSpec(35, g, g, 128, round_half_even(0.05 * nv), 3,
                                 keep_for_ratio(nv, 0.11) if keep is None else keep))
        return Spec("highres-sweep", 4, 4, 32, 32, 4096, ims)
    raise ValueError(f"unknown config {cfg}")


@dataclasses.dataclass
class Inputs:
    spec: Spec
    n_sys: np.ndarray
    n_vis: np.ndarray
    n_text: np.ndarray
    grid_h: np.ndarray
    grid_w: np.ndarray
    tok_off: np.ndarray
    vis_off: np.ndarray
    text_off: np.ndarray
    keep: np.ndarray          # [B] K per image
    keep_off: np.ndarray      # [B+1]
    q_text: np.ndarray        # uint16 [L, sum_text, H, d]
    k: np.ndarray             # uint16 [L, sum_T, H_kv, d]
    v: Optional[np.ndarray]   # uint16 [L, sum_T, H_kv, d]
    hidden: Optional[np.ndarray]  # uint16 [sum_T, D]
    salient: List[np.ndarray]     # per image: sorted visual indices


def _salient_positions(rng: np.random.Generator, h: int, w: int, n: int, blobs: int) -> np.ndarray:
    n = min(n, h * w)
    if n <= 0:
        return np.zeros(0, dtype=np.int64)
    if blobs <= 0:
        return np.sort(rng.choice(h * w, size=n, replace=False))
    ii, jj = np.meshgrid(np.arange(h), np.arange(w), indexing="ij")
    pts = np.stack([ii.ravel(), jj.ravel()], axis=1).astype(np.float64)
    centres = rng.uniform([0, 0], [h - 1, w - 1], size=(blobs, 2))
    sizes = [n // blobs + (1 if b < n % blobs else 0) for b in range(blobs)]
    taken = np.zeros(h * w, dtype=bool)
    for c, s in zip(centres, sizes):
        dist = ((pts - c) ** 2).sum(axis=1)
        dist[taken] = np.inf
        order = np.argsort(dist, kind="stable")[:s]
        taken[order] = True
    return np.nonzero(taken)[0]


def make_inputs(spec: Spec, *, with_payload: bool = True) -> Inputs:
    """Draw every tensor of one batch.  ``with_payload`` adds V and hidden."""
    B, L, H, Hkv, d = spec.B, spec.L, spec.H, spec.H_kv, spec.d
    if H % Hkv:
        raise ValueError("H must be a multiple of H_kv")
    group = H // Hkv
    n_sys = np.array([im.n_sys for im in spec.images], dtype=np.int32)
    n_vis = np.array([im.n_vis for im in spec.images], dtype=np.int32)
    n_text = np.array([im.n_text for im in spec.images], dtype=np.int32)
    grid_h = np.array([im.grid_h for im in spec.images], dtype=np.int32)
    grid_w = np.array([im.grid_w for im in spec.images], dtype=np.int32)
    T = n_sys + n_vis + n_text
    tok_off = np.concatenate([[0], np.cumsum(T)]).astype(np.int32)
    vis_off = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int32)
    text_off = np.concatenate([[0], np.cumsum(n_text)]).astype(np.int32)
    keep = np.array([im.keep for im in spec.images], dtype=np.int32)
    keep_off = np.concatenate([[0], np.cumsum(keep)]).astype(np.int32)
    sum_T, sum_text = int(tok_off[-1]), int(text_off[-1])

    q = np.empty((L, sum_text, H, d), dtype=np.uint16)
    k = np.empty((L, sum_T, Hkv, d), dtype=np.uint16)
    payload = with_payload and spec.hidden > 0
    v = np.empty((L, sum_T, Hkv, d), dtype=np.uint16) if payload else None
    hid = np.empty((sum_T, spec.hidden), dtype=np.uint16) if payload else None
    amp = SIGMA * np.sqrt(d)

    def draw_image(b: int) -> np.ndarray:
        im = spec.images[b]
        rng = np.random.Generator(np.random.PCG64(1000 * spec.cfg_id + b))
        # V and the hidden states come from a stream of their own, so Q and K
        # are the same with or without the payload
        prng = np.random.Generator(np.random.PCG64(1000 * spec.cfg_id + b + (1 << 40)))
        sal = _salient_positions(rng, im.grid_h, im.grid_w, im.n_salient, im.blobs)
        t0, t1 = int(tok_off[b]), int(tok_off[b + 1])
        x0, x1 = int(text_off[b]), int(text_off[b + 1])
        for l in range(L):
            kk = rng.standard_normal((t1 - t0, Hkv, d), dtype=np.float32) * np.float32(SIGMA)
            qq = rng.standard_normal((x1 - x0, H, d), dtype=np.float32) * np.float32(SIGMA)
            u = rng.standard_normal((Hkv, d)).astype(np.float64)
            u /= np.linalg.norm(u, axis=1, keepdims=True)
            g = rng.uniform(0.0, 1.5, size=H)
            if sal.size:
                kk[im.n_sys + sal] += (4.0 * amp * u).astype(np.float32)[None]
            qq += (g[:, None] * amp * u[np.arange(H) // group]).astype(np.float32)[None]
            k[l, t0:t1] = bf16_bits(kk)
            q[l, x0:x1] = bf16_bits(qq)
            if payload:
                v[l, t0:t1] = bf16_bits(prng.standard_normal((t1 - t0, Hkv, d), dtype=np.float32))
        if payload:
            hid[t0:t1] = bf16_bits(prng.standard_normal((t1 - t0, spec.hidden), dtype=np.float32))
        return sal

    # Images draw from streams of their own and write disjoint rows, so they
    # run on a thread pool (numpy releases the GIL while it fills the arrays);
    # the values do not depend on the number of threads.
    workers = max(1, min(B, os.cpu_count() or 1, 16))
    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        salient = list(ex.map(draw_image, range(B)))
    return Inputs(spec, n_sys, n_vis, n_text, grid_h, grid_w, tok_off, vis_off, text_off,
                  keep, keep_off, q, k, v, hid, salient)


def full_queries(inp: Inputs) -> np.ndarray:
    """Queries of every row of every image, [L, sum T, H, d] bf16 bits, for the
    layer's own attention pass: the text rows are inp.q_text (so the text
    rows' scores are those of the decision), the system and visual rows are
    i.i.d. normal with variance d**-0.5 from a stream of their own per image
    (seed 1000 * config + image + 2**41)."""
    s = inp.spec
    q = np.empty((s.L, int(inp.tok_off[-1]), s.H, s.d), dtype=np.uint16)
    for b in range(s.B):
        rng = np.random.Generator(np.random.PCG64(1000 * s.cfg_id + b + (1 << 41)))
        t0, S, NV, NT = int(inp.tok_off[b]), int(inp.n_sys[b]), int(inp.n_vis[b]), int(inp.n_text[b])
        x0 = int(inp.text_off[b])
        for l in range(s.L):
            q[l, t0:t0 + S + NV] = bf16_bits(
                rng.standard_normal((S + NV, s.H, s.d), dtype=np.float32) * np.float32(SIGMA))
            q[l, t0 + S + NV:t0 + S + NV + NT] = inp.q_text[l, x0:x0 + NT]
    return q


def custom_spec(name: str, images: Sequence[ImageSpec], *, L: int = 2, H: int = 4, H_kv: int = 4,
                hidden: int = 0, cfg_id: int = 9) -> Spec:
    """A free-form spec for edge-case tests (small heads, odd grids, K=0 ...)."""
    return Spec(name, cfg_id, L, H, H_kv, hidden, list(images))
