"""Host-side logic: input generator and budget schedules (no GPU)."""
import json
import os

import numpy as np
import pytest
import torch

from paper_2608_23253_gb300 import budget, synth
from tests.conftest import GOLDEN


def test_avg_tokens_printed_schedules():
    g = json.load(open(os.path.join(GOLDEN, "avg_tokens_schedules.json")))
    for s in g["schedules"]:
        got = budget.avg_tokens(g["n_layers"], g["n_visual"], g["prune_after"], s["keep"])
        assert got == s["avg"], s


def test_avg_tokens_layer_spans():
    t = budget.tokens_per_layer(32, 576, [3, 17, 22], [122, 48, 42])
    assert t[:3] == [576] * 3 and t[3:17] == [122] * 14 and t[17:22] == [48] * 5 and t[22:] == [42] * 10


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).normal(size=100000).astype(np.float32) * 7
    x[:4] = [0.0, -0.0, 1.00390625, 1.01171875]      # exact ties to even
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(synth.bf16_bits(x), want)
    assert np.array_equal(synth.bf16_to_f32(want), torch.from_numpy(want.view(np.int16)).view(
        torch.bfloat16).float().numpy())


@pytest.mark.parametrize("cfg", [0, 1, 2, 3, 4])
def test_config_shapes(cfg):
    spec = synth.config_spec(cfg)
    if cfg == 0:
        assert (spec.B, spec.L, spec.H, spec.images[0].n_text, spec.images[0].keep) == (1, 2, 32, 32, 64)
    if cfg == 1:
        assert (spec.B, spec.L, spec.hidden, spec.images[0].n_tok) == (1, 3, 4096, 675)
    if cfg == 2:
        nts = [im.n_text for im in spec.images]
        assert spec.B == 32 and min(nts) >= 16 and max(nts) <= 128 and len(set(nts)) > 5
    if cfg == 3:
        assert (spec.H, spec.H_kv, spec.B) == (28, 4, 16)
        for im in spec.images:
            assert (im.grid_h, im.grid_w) in [(16, 16), (24, 32), (32, 32), (36, 36)]
            assert im.keep == {256: 28, 768: 85, 1024: 114, 1296: 144}[im.n_vis]
    if cfg == 4:
        assert {im.n_vis: im.keep for im in spec.images} == {2304: 253, 4096: 451}
        assert {im.n_vis: im.n_salient for im in spec.images} == {2304: 115, 4096: 205}


@pytest.mark.parametrize("ratio", [1 / 3, 2 / 9])
def test_qwen2vl_dynamic_grid_spec(ratio):
    """Sec. 4.5's reduction ratios on merged-patch grids of any shape."""
    spec = synth.config_spec(3, keep_ratio=ratio, dynamic_grids=True)
    again = synth.config_spec(3, keep_ratio=ratio, dynamic_grids=True)
    assert [(i.grid_h, i.grid_w) for i in spec.images] == \
        [(i.grid_h, i.grid_w) for i in again.images]
    assert (spec.B, spec.H, spec.H_kv, spec.L) == (16, 28, 4, 3)
    for im in spec.images:
        assert 12 <= im.grid_h <= 48 and 12 <= im.grid_w <= 48 and im.n_vis <= 1296
        assert im.keep == int(np.round(ratio * im.n_vis))
        assert im.n_text == 64
    assert any(im.grid_h % 4 or im.grid_w % 4 for im in spec.images)
    # the fixed-grid configuration is unchanged by the new options' defaults
    assert [(i.grid_h, i.grid_w, i.keep) for i in synth.config_spec(3).images] == \
        [(i.grid_h, i.grid_w, i.keep) for i in synth.config_spec(3, keep_ratio=None).images]


def test_generator_deterministic_and_planted():
    spec = synth.config_spec(1)
    a = synth.make_inputs(spec, with_payload=False)
    b = synth.make_inputs(spec, with_payload=False)
    assert np.array_equal(a.k, b.k) and np.array_equal(a.q_text, b.q_text)
    assert a.salient[0].size == 40
    assert a.k.shape == (3, 675, 32, 128) and a.q_text.shape == (3, 64, 32, 128)
    k = synth.bf16_to_f32(a.k[0, :, 0]).astype(np.float64)
    norms = np.linalg.norm(k, axis=1)
    sal = 35 + a.salient[0]
    others = np.setdiff1d(np.arange(35, 611), sal)
    assert norms[sal].mean() > 3 * norms[others].mean()


def test_payload_does_not_change_q_and_k():
    """V and the hidden states come from their own stream: a test that needs the
    payload may reuse the oracle computed on the inputs without it."""
    spec = synth.config_spec(0)
    spec.hidden = 64
    a = synth.make_inputs(spec, with_payload=True)
    b = synth.make_inputs(spec, with_payload=False)
    assert np.array_equal(a.k, b.k) and np.array_equal(a.q_text, b.q_text)
    assert a.v is not None and b.v is None and a.hidden.shape == (643, 64)


def test_blobs_are_spatially_clustered():
    spec = synth.config_spec(1)
    inp = synth.make_inputs(spec, with_payload=False)
    s = inp.salient[0]
    i, j = s // 24, s % 24
    # 40 points in 3 blobs: the mean nearest-neighbour distance is ~1 grid step
    d = np.sqrt((i[:, None] - i[None]) ** 2 + (j[:, None] - j[None]) ** 2) + np.eye(s.size) * 99
    assert d.min(axis=1).mean() < 1.5


def test_multiply_high_division_is_exact():
    """The cell arithmetic of the select divides small non-negative ints by 2 <= d <= 2^13 as
    umulhi(n, ceil(2^32 / d)) (d = 1 takes a plain division: its multiplier
    does not fit 32 bits); the claim is exactness for every n < 2^17.
    Checked at the worst numerators n = q*d + d - 1 (largest fractional part)
    and at the multiples n = q*d, for every d."""
    import numpy as np
    for d in range(2, 8193):
        assert ((1 << 32) + d - 1) // d < (1 << 32)
        m = ((1 << 32) + d - 1) // d
        q = np.arange(0, (1 << 17) // d + 1, dtype=np.uint64)
        for n in (q * np.uint64(d), q * np.uint64(d) + np.uint64(d - 1)):
            n = n[n < (1 << 17)]
            got = (n * np.uint64(m)) >> np.uint64(32)
            assert np.array_equal(got, n // np.uint64(d)), d


def test_bench_attention_lse_matches_oracle():
    """bench.py's stand-in for the attention pass's row lse (torch, float32)
    against the oracle's float64 causal_row_lse, on the CPU."""
    import bench
    from oracle import e2s_oracle as orc
    inp = synth.make_inputs(synth.custom_spec(
        "lse", [synth.ImageSpec(35, 12, 12, 20, 10, 2, 30),
                synth.ImageSpec(3, 5, 7, 9, 4, 0, 10)], L=2, H=8, H_kv=2, cfg_id=94),
        with_payload=False)
    q = torch.from_numpy(inp.q_text.view(np.int16)).view(torch.bfloat16)
    k = torch.from_numpy(inp.k.view(np.int16)).view(torch.bfloat16)
    got = bench.attention_lse(inp, q, k, torch.device("cpu")).numpy()
    want = orc.text_row_lse(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text, H_kv=2)
    assert got.shape == want.shape
    assert np.abs(got - want).max() < 1e-4


def test_bench_ablation_flags_parse_to_the_header_values():
    """bench --flags: Table 2's A1..A5 names map to the E2S_* flag bits."""
    import bench
    assert bench.parse_flags("") == 0
    assert bench.parse_flags("A1") == 16 and bench.parse_flags("a2") == 1
    assert bench.parse_flags("A3,A4") == 2 | 4 and bench.parse_flags("A5") == 8
    assert bench.parse_flags("0x6") == 6
    assert {v[1] for v in bench.ABLATIONS.values()} == {1, 2, 4, 8, 16}
