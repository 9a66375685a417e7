"""Shared GPU-test plumbing: run the CUDA path and the oracle on the same inputs."""
from __future__ import annotations

import functools

import numpy as np
import torch

from oracle import e2s_oracle as orc
from paper_2608_23253_gb300 import synth

MODES = {"causal": (1, orc.SCORE_CAUSAL_PROB), "eq1": (0, orc.SCORE_EQ1)}


def device():
    if not torch.cuda.is_available():
        raise RuntimeError("GPU tests need CUDA")
    return torch.device("cuda:0")


PATHS = ("decide", "fuse_select", "separate")


def run_gpu(inp, mode: str = "causal", *, simt: bool = False, flags: int = 0, lam: float = 0.1,
            G: int = 4, keep=None, norm_mode: int = 0, prior=None, cand=None,
            grid_h=None, grid_w=None, path: str = "decide"):
    """The decision through one of the ABI call sequences:
    decide       e2s_decide (score, then token-parallel evidence + select)
    fuse_select  e2s_score, then e2s_fuse_select (one cluster per image)
    separate     e2s_score, e2s_fuse, e2s_select"""
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    dev = device()
    s = inp.spec
    gh = inp.grid_h if grid_h is None else grid_h
    gw = inp.grid_w if grid_w is None else grid_w
    batch = Batch(inp.n_sys, inp.n_vis, inp.n_text, gh, gw, L=s.L, H=s.H, H_kv=s.H_kv, device=dev)
    f = flags | (e2s.E2S_SIMT_SCORE if simt else 0)
    par = e2s.params(lam=lam, G=G, score_mode=MODES[mode][0], norm_mode=norm_mode, flags=f)
    dec = Decision(batch, inp.keep if keep is None else keep, par)
    q = bf16_tensor(inp.q_text, dev)
    k = bf16_tensor(inp.k, dev)
    pr = None if prior is None else torch.as_tensor(
        np.concatenate([prior, np.zeros((prior.shape[0], 1))], axis=1).astype(np.float32),
        device=dev)
    cd = None if cand is None else torch.as_tensor(np.concatenate(cand).astype(np.int32),
                                                   device=dev)
    if path == "decide":
        dec.decide(q, k, prior=pr, cand=cd)
    elif path == "fuse_select":
        dec.score(q, k)
        dec.fuse_select(prior=pr, cand=cd)
    elif path == "separate":
        dec.score(q, k)
        dec.fuse(prior=pr)
        dec.select(cand=cd)
    else:
        raise ValueError(path)
    torch.cuda.synchronize()
    st = dec.status()
    out = {
        "a": dec.a.cpu().numpy(), "mass": dec.mass.cpu().numpy(), "fused": dec.fused.cpu().numpy(),
        "q": dec.q.cpu().numpy(), "q_tilde": dec.q_tilde.cpu().numpy(), "keep": dec.keep_lists(),
        "status": st, "decision": dec, "q_dev": q, "k_dev": k,
    }
    return out


def run_oracle(inp, mode: str = "causal", *, flags: int = 0, lam: float = 0.1, G: int = 4,
               keep=None, norm=None, prior=None, cand=None, grid_h=None, grid_w=None):
    p = orc.Params(lam=lam, G=G, score_mode=MODES[mode][1], norm_mode=norm, flags=flags)
    out = orc.decide(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text,
                      inp.grid_h if grid_h is None else grid_h,
                      inp.grid_w if grid_w is None else grid_w,
                      inp.keep if keep is None else keep, H_kv=inp.spec.H_kv, params=p,
                      prior=prior, cand=cand)
    out["score_mode"] = p.score_mode
    return out


@functools.lru_cache(maxsize=None)
def config_inputs(cfg: int, batch=None, keep=None, payload=False):
    return synth.make_inputs(synth.config_spec(cfg, batch=batch, keep=keep), with_payload=payload)


@functools.lru_cache(maxsize=None)
def config_oracle(cfg: int, batch, keep, mode: str):
    return run_oracle(config_inputs(cfg, batch, keep), mode)
