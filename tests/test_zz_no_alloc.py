"""e2s_fuse_noalloc: the workspace-free variant of e2s_fuse (GPU).

Callers that cannot allocate device memory (a host framework that owns the
device heap, an FFI plug-in without an allocator, a real-time loop that bans
cudaMalloc) use this entry point; its scratch lives in a static device array
inside the library.  Here it is called through the C ABI twice in a row, on
two different batches, and each result is compared with e2s_fuse on the same
inputs.  The file name sorts last so that a run stopping at the first failure
has already run every other test; it also passes alone in a fresh process.
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
