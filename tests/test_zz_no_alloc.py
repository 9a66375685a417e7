"""e2s_fuse_noalloc: the workspace-free variant of e2s_fuse (GPU).

Callers that cannot allocate device memory (a host framework that owns the
device heap, an FFI plug-in without an allocator, a real-time loop that bans
cudaMalloc) use this entry point; its scratch lives in a static device array
inside the library.  Here it is called through the C ABI twice in a row, on
two different batches, and each result is compared with e2s_fuse on the same
inputs; then, over the ablation flags, the softmax normalisation, a carried
prior and a missing mass output, with the float64 oracle directly.  The file
name sorts last so that a run stopping at the first failure has already run
every other test; it also passes alone in a fresh process.
"""
import numpy as np
import pytest
import torch

from tests import parity
from tests.gpu_helpers import config_inputs, device

pytestmark = pytest.mark.gpu


def _fuse_both(inp):
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    dev = device()
    batch = Batch.from_inputs(inp, device=dev)
    dec = Decision(batch, inp.keep, e2s.params())
    dec.score(bf16_tensor(inp.q_text, dev), bf16_tensor(inp.k, dev))
    dec.fuse()
    V = batch.sum_vis
    mass = torch.full((batch.L, V, 4), np.nan, dtype=torch.float32, device=dev)
    fused = torch.full((V, 4), np.nan, dtype=torch.float32, device=dev)
    q = torch.full((V,), np.nan, dtype=torch.float32, device=dev)
    st = e2s.e2s_fuse_noalloc(batch.layout, dec.params, dec.a, None, None, mass, fused, q, None)
    assert st == e2s.E2S_OK, e2s.e2s_status_string(st)
    torch.cuda.synchronize()
    assert dec.status() == e2s.E2S_OK
    return dec, mass.cpu().numpy(), fused.cpu().numpy(), q.cpu().numpy()


def test_noalloc_matches_fuse_on_two_calls_in_a_row():
    for cfg, batch in ((2, 4), (0, None)):           # a larger batch first, then a smaller one
        inp = config_inputs(cfg, batch, None)
        dec, mass, fused, q = _fuse_both(inp)
        parity.assert_close("mass", mass, dec.mass.cpu().numpy())
        parity.assert_close("fused", fused, dec.fused.cpu().numpy())
        parity.assert_close("q", q, dec.q.cpu().numpy())


def test_noalloc_rejects_batches_beyond_its_capacity():
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch
    dev = device()
    B = 86                                            # 86 * 3 * 32 = 8256 > 8192
    batch = Batch([35] * B, [4] * B, [2] * B, [2] * B, [2] * B, L=3, H=32, H_kv=32, device=dev)
    out = torch.zeros((batch.sum_vis, 4), dtype=torch.float32, device=dev)
    st = e2s.e2s_fuse_noalloc(batch.layout, e2s.params(), out, None, None, None, out, out, None)
    assert st == e2s.E2S_ERR_WORKSPACE


_VARIANTS = {
    "default": dict(flags=0, norm=None, prior=False, mass=True),
    "prior": dict(flags=0, norm=None, prior=True, mass=True),
    "softmax-norm": dict(flags=0, norm="softmax", prior=False, mass=True),
    "no-reliability": dict(flags=1, norm=None, prior=False, mass=True),
    "no-layer-fusion+prior": dict(flags=2, norm=None, prior=True, mass=True),
    "no-conflict": dict(flags=4, norm=None, prior=False, mass=True),
    "vanilla": dict(flags=16, norm=None, prior=False, mass=True),
    "no-mass-out": dict(flags=0, norm=None, prior=True, mass=False),
}


@pytest.mark.parametrize("variant", sorted(_VARIANTS))
@pytest.mark.parametrize("cfg,batch", [(0, None), (2, 3)])
def test_noalloc_matches_oracle(variant, cfg, batch):
    """Masses, fused masses, conflict and q against the float64 oracle, with
    the same options given to e2s_fuse for comparison."""
    from oracle import e2s_oracle as orc
    from paper_2608_23253_gb300 import e2s
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor
    from tests.gpu_helpers import run_oracle
    v = _VARIANTS[variant]
    dev = device()
    inp = config_inputs(cfg, batch, None)
    V = int(inp.vis_off[-1])
    prior = None
    if v["prior"]:
        prior = np.random.default_rng(77).dirichlet([2.0, 1.0, 1.0], size=V)
    ref = run_oracle(inp, "causal", flags=v["flags"], norm=v["norm"], prior=prior)
    norm_mode = e2s.E2S_NORM_SOFTMAX if v["norm"] == orc.NORM_SOFTMAX else e2s.E2S_NORM_DEFAULT
    batch_ = Batch.from_inputs(inp, device=dev)
    dec = Decision(batch_, inp.keep, e2s.params(flags=v["flags"], norm_mode=norm_mode))
    dec.score(bf16_tensor(inp.q_text, dev), bf16_tensor(inp.k, dev))
    pr = None if prior is None else torch.as_tensor(
        np.concatenate([prior, np.zeros((V, 1))], axis=1).astype(np.float32), device=dev)
    dec.fuse(prior=pr)
    mass = torch.full((batch_.L, V, 4), np.nan, dtype=torch.float32, device=dev) if v["mass"] else None
    fused = torch.full((V, 4), np.nan, dtype=torch.float32, device=dev)
    q = torch.full((V,), np.nan, dtype=torch.float32, device=dev)
    st = e2s.e2s_fuse_noalloc(batch_.layout, dec.params, dec.a, None, pr, mass, fused, q, None)
    assert st == e2s.E2S_OK, e2s.e2s_status_string(st)
    torch.cuda.synchronize()
    assert dec.status() == e2s.E2S_OK
    f, qq = fused.cpu().numpy(), q.cpu().numpy()
    parity.check_a(dec.a.cpu().numpy(), ref["a"], causal=True)
    if mass is not None:
        m = mass.cpu().numpy()
        parity.assert_close("mass", m[..., :3], ref["mass"])
        parity.assert_close("p_bar", m[..., 3], ref["p_bar"])
        parity.assert_close("mass vs e2s_fuse", m, dec.mass.cpu().numpy())
    parity.assert_close("fused", f[:, :3], ref["fused"])
    parity.assert_close("K", f[:, 3], ref["K"])
    parity.assert_close("q", qq, ref["q"])
    parity.assert_close("fused vs e2s_fuse", f, dec.fused.cpu().numpy())
    parity.assert_close("q vs e2s_fuse", qq, dec.q.cpu().numpy())
