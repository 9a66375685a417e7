"""Buffers and call sequence of one pruning decision, on top of the C ABI.

PyTorch provides device memory and streams only; every step of the decision
runs in libe2s.so kernels:

    score  -> a[L][H][sum_vis]            (Sec. 3.1 Eq. 1 / causal-prefix probability)
    fuse   -> mass, fused (I,U,Theta,K), q (Sec. 4.1-4.2, Eqs. 8-19)
    select -> q~, keep_idx                (Sec. 4.3, Eqs. 20-23)
    compact-> shortened hidden / K / V    (the next layer's input)

decide() runs score, fuse and select through e2s_decide (two launches);
prune() adds the compaction (e2s_prune, three launches).
"""
from __future__ import annotations

from typing import Optional, Sequence

import numpy as np
import torch

from . import e2s


def _i32(x, device) -> torch.Tensor:
    return torch.as_tensor(np.asarray(x, dtype=np.int32), device=device)


def bf16_tensor(bits: np.ndarray, device) -> torch.Tensor:
    """uint16 bf16 bit patterns -> torch.bfloat16 tensor on `device` (same bytes)."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.view(torch.bfloat16).to(device)


class Batch:
    """Device-side layout of a packed batch: [system][visual h x w][text] per image."""

    def __init__(self, n_sys, n_vis, n_text, grid_h, grid_w, *, L: int, H: int, H_kv: int,
                 d: int = 128, device="cuda"):
        n_sys, n_vis, n_text = (np.asarray(x, dtype=np.int64) for x in (n_sys, n_vis, n_text))
        T = n_sys + n_vis + n_text
        self.B, self.L, self.H, self.H_kv, self.d = len(n_vis), L, H, H_kv, d
        self.n_sys_h, self.n_vis_h, self.n_text_h = n_sys, n_vis, n_text
        self.tok_off_h = np.concatenate([[0], np.cumsum(T)]).astype(np.int64)
        self.vis_off_h = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int64)
        self.text_off_h = np.concatenate([[0], np.cumsum(n_text)]).astype(np.int64)
        self.device = device
        self._arrays = {
            "tok_off": _i32(self.tok_off_h, device), "n_sys": _i32(n_sys, device),
            "n_vis": _i32(n_vis, device), "n_text": _i32(n_text, device),
            "grid_h": _i32(grid_h, device), "grid_w": _i32(grid_w, device),
            "vis_off": _i32(self.vis_off_h, device), "text_off": _i32(self.text_off_h, device),
        }
        a = self._arrays
        self.sum_T, self.sum_vis, self.sum_text = int(T.sum()), int(n_vis.sum()), int(n_text.sum())
        self.layout = e2s.e2s_layout(
            self.B, L, H, H_kv, d,
            a["tok_off"].data_ptr(), a["n_sys"].data_ptr(), a["n_vis"].data_ptr(),
            a["n_text"].data_ptr(), a["grid_h"].data_ptr(), a["grid_w"].data_ptr(),
            a["vis_off"].data_ptr(), a["text_off"].data_ptr(),
            int(T.max()), int(n_vis.max()), int(n_text.max()),
            self.sum_T, self.sum_vis, self.sum_text)

    @classmethod
    def from_inputs(cls, inp, device="cuda") -> "Batch":
        s = inp.spec
        return cls(inp.n_sys, inp.n_vis, inp.n_text, inp.grid_h, inp.grid_w, L=s.L, H=s.H,
                   H_kv=s.H_kv, d=s.d, device=device)

    def array(self, name: str) -> torch.Tensor:
        return self._arrays[name]


class Decision:
    """Output buffers, workspace and the four ABI calls of one decision."""

    def __init__(self, batch: Batch, keep_counts: Sequence[int], params: e2s.e2s_params, *,
                 with_mass: bool = True, with_q_tilde: bool = True):
        dev = batch.device
        self.batch, self.params = batch, params
        L, H, V = batch.L, batch.H, batch.sum_vis
        f32 = dict(dtype=torch.float32, device=dev)
        self.a = torch.zeros((L, H, V), **f32)
        self.mass = torch.zeros((L, V, 4), **f32) if with_mass else None
        self.fused = torch.zeros((V, 4), **f32)
        self.q = torch.zeros(V, **f32)
        self.q_tilde = torch.zeros(V, **f32) if with_q_tilde else None
        kc = np.asarray(keep_counts, dtype=np.int64)
        self.keep_counts_h = kc
        self.keep_off_h = np.concatenate([[0], np.cumsum(kc)]).astype(np.int64)
        self.sum_keep = int(self.keep_off_h[-1])
        self.keep_count = _i32(kc, dev)
        self.keep_off = _i32(self.keep_off_h, dev)
        self.keep_idx = torch.full((max(self.sum_keep, 1),), -1, dtype=torch.int32, device=dev)
        self.ws_bytes = e2s.e2s_workspace_size(batch.layout, params)
        if self.ws_bytes == 0:
            raise e2s.E2SError(e2s.E2S_ERR_SHAPE, "e2s_workspace_size")
        self.ws = torch.zeros(self.ws_bytes, dtype=torch.uint8, device=dev)

    # -- the four ABI calls
    def score(self, q_text: torch.Tensor, k: torch.Tensor, stream=None,
              q_row_stride: Optional[int] = None, k_row_stride: Optional[int] = None,
              lse: Optional[torch.Tensor] = None) -> None:
        """e2s_score, or e2s_score_lse when the text rows' attention lse is given."""
        b = self.batch
        qs = q_row_stride if q_row_stride is not None else b.H * b.d
        ks = k_row_stride if k_row_stride is not None else b.H_kv * b.d
        if lse is not None:
            e2s.check(e2s.e2s_score_lse(b.layout, self.params, q_text, qs, k, ks, lse, self.a,
                                        self.ws, self.ws_bytes, stream), "e2s_score_lse")
            return
        e2s.check(e2s.e2s_score(b.layout, self.params, q_text, qs, k, ks, self.a, self.ws,
                                self.ws_bytes, stream), "e2s_score")

    def fuse(self, prior: Optional[torch.Tensor] = None, cand: Optional[torch.Tensor] = None,
             stream=None) -> None:
        e2s.check(e2s.e2s_fuse(self.batch.layout, self.params, self.a, cand, prior, self.mass,
                               self.fused, self.q, self.ws, self.ws_bytes, stream), "e2s_fuse")

    def fuse_select(self, prior: Optional[torch.Tensor] = None,
                    cand: Optional[torch.Tensor] = None, stream=None) -> None:
        """fuse + select in one launch (same results as the two calls)."""
        e2s.check(e2s.e2s_fuse_select(self.batch.layout, self.params, self.a, cand, prior,
                                      self.mass, self.fused, self.q, self.keep_count,
                                      self.keep_off, self.sum_keep, self.keep_idx, self.q_tilde,
                                      self.ws, self.ws_bytes, stream), "e2s_fuse_select")

    def select(self, cand: Optional[torch.Tensor] = None, stream=None) -> None:
        e2s.check(e2s.e2s_select(self.batch.layout, self.params, self.q, cand, self.keep_count,
                                 self.keep_off, self.sum_keep, self.keep_idx, self.q_tilde,
                                 self.ws, self.ws_bytes, stream), "e2s_select")

    def out_rows(self) -> int:
        return self.batch.sum_T - self.batch.sum_vis + self.sum_keep

    def compact(self, src: Sequence[torch.Tensor], dst: Sequence[torch.Tensor],
                pos_ids: Optional[torch.Tensor] = None, stream=None) -> None:
        row_bytes = [t.stride(0) * t.element_size() for t in src]
        e2s.check(e2s.e2s_compact(self.batch.layout, self.keep_idx, self.keep_off, self.sum_keep,
                                  len(src), src, dst, row_bytes, pos_ids, self.ws, self.ws_bytes,
                                  stream), "e2s_compact")

    def decide(self, q_text: torch.Tensor, k: torch.Tensor, prior: Optional[torch.Tensor] = None,
               cand: Optional[torch.Tensor] = None, stream=None,
               q_row_stride: Optional[int] = None, k_row_stride: Optional[int] = None,
               lse: Optional[torch.Tensor] = None) -> None:
        """score + fuse + select in two launches (e2s_decide; e2s_decide_lse when
        the text rows' attention lse is given)."""
        b = self.batch
        qs = q_row_stride if q_row_stride is not None else b.H * b.d
        ks = k_row_stride if k_row_stride is not None else b.H_kv * b.d
        if lse is not None:
            e2s.check(e2s.e2s_decide_lse(b.layout, self.params, q_text, qs, k, ks, lse, cand,
                                         prior, self.a, self.mass, self.fused, self.q,
                                         self.keep_count, self.keep_off, self.sum_keep,
                                         self.keep_idx, self.q_tilde, self.ws, self.ws_bytes,
                                         stream), "e2s_decide_lse")
            return
        e2s.check(e2s.e2s_decide(b.layout, self.params, q_text, qs, k, ks, cand, prior, self.a,
                                 self.mass, self.fused, self.q, self.keep_count, self.keep_off,
                                 self.sum_keep, self.keep_idx, self.q_tilde, self.ws,
                                 self.ws_bytes, stream), "e2s_decide")

    def prune(self, q_text: torch.Tensor, k: torch.Tensor, src: Sequence[torch.Tensor],
              dst: Sequence[torch.Tensor], pos_ids: Optional[torch.Tensor] = None,
              prior: Optional[torch.Tensor] = None, cand: Optional[torch.Tensor] = None,
              stream=None, lse: Optional[torch.Tensor] = None) -> None:
        """The whole pruning step (e2s_prune): decide, then compact src into dst
        (e2s_prune_lse when the text rows' attention lse is given)."""
        b = self.batch
        row_bytes = [t.stride(0) * t.element_size() for t in src]
        if lse is not None:
            e2s.check(e2s.e2s_prune_lse(b.layout, self.params, q_text, b.H * b.d, k,
                                        b.H_kv * b.d, lse, cand, prior, self.a, self.mass,
                                        self.fused, self.q, self.keep_count, self.keep_off,
                                        self.sum_keep, self.keep_idx, self.q_tilde, len(src), src,
                                        dst, row_bytes, pos_ids, self.ws, self.ws_bytes, stream),
                      "e2s_prune_lse")
            return
        e2s.check(e2s.e2s_prune(b.layout, self.params, q_text, b.H * b.d, k, b.H_kv * b.d, cand,
                                prior, self.a, self.mass, self.fused, self.q, self.keep_count,
                                self.keep_off, self.sum_keep, self.keep_idx, self.q_tilde,
                                len(src), src, dst, row_bytes, pos_ids, self.ws, self.ws_bytes,
                                stream), "e2s_prune")

    def attention(self, q_all: torch.Tensor, k: torch.Tensor, v: torch.Tensor,
                  o_out: torch.Tensor, lse_out: Optional[torch.Tensor] = None,
                  with_score: bool = True, stream=None) -> None:
        """e2s_attention: the layer's causal attention over q_all [L, sum_T, H, d]
        (every row), into o_out (same shape) and lse_out [L, H, sum_T]; with
        with_score, the decision's score into self.a as a by-product."""
        b = self.batch
        e2s.check(e2s.e2s_attention(b.layout, q_all, b.H * b.d, k, b.H_kv * b.d, v,
                                    b.H_kv * b.d, o_out, b.H * b.d, lse_out,
                                    self.a if with_score else None, self.ws, self.ws_bytes,
                                    stream), "e2s_attention")

    def decide_attn(self, q_all: torch.Tensor, k: torch.Tensor, v: torch.Tensor,
                    o_out: torch.Tensor, lse_out: Optional[torch.Tensor] = None,
                    prior: Optional[torch.Tensor] = None, cand: Optional[torch.Tensor] = None,
                    stream=None) -> None:
        """e2s_decide_attn: the layer's attention, then the decision from its score."""
        b = self.batch
        e2s.check(e2s.e2s_decide_attn(b.layout, self.params, q_all, b.H * b.d, k, b.H_kv * b.d,
                                      v, b.H_kv * b.d, o_out, b.H * b.d, lse_out, cand, prior,
                                      self.a, self.mass, self.fused, self.q, self.keep_count,
                                      self.keep_off, self.sum_keep, self.keep_idx, self.q_tilde,
                                      self.ws, self.ws_bytes, stream), "e2s_decide_attn")

    def run(self, q_text: torch.Tensor, k: torch.Tensor, stream=None) -> None:
        """The decision itself: score + fuse + select (e2s_decide)."""
        self.decide(q_text, k, stream=stream)

    def status(self, stream=None) -> int:
        return e2s.e2s_read_status(self.ws, stream)

    def keep_lists(self):
        idx = self.keep_idx.cpu().numpy()
        return [idx[self.keep_off_h[b]:self.keep_off_h[b + 1]] for b in range(self.batch.B)]
