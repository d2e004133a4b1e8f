"""CPU checks of the seeded input generators."""
import numpy as np
import torch

from paper_2602_06161_gb300 import workloads as W


def test_bf16_rounding_matches_torch_rne():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 7,
                        np.array([1.00390625, 1.01171875, -2.0078125, 0.0, -0.0, 3.0e38], np.float32)])
    ours = W.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    back = W.bf16_bits_to_f32(ours)
    assert np.array_equal(back, torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_attn_inputs_deterministic_and_seeds_valid():
    a = W.make_attn_inputs(2, 4, 2, 300, 16, 9, dtype="bf16", seed=3, seed_lo=100, seed_hi=300)
    b = W.make_attn_inputs(2, 4, 2, 300, 16, 9, dtype="bf16", seed=3, seed_lo=100, seed_hi=300)
    for name in ["q", "k_cached", "v_cached", "k_seedmask", "v_seedmask", "seed_idx"]:
        assert np.array_equal(getattr(a, name), getattr(b, name))
    assert a.q.dtype == np.uint16 and a.q.shape == (2, 4, 300, 16)
    assert a.k_seedmask.shape == (2, 2, 9, 16)
    for row in a.seed_idx:
        assert len(set(row.tolist())) == 9
        assert row.min() >= 100 and row.max() < 300


def test_runs_placement_disjoint():
    inp = W.make_attn_inputs(3, 2, 2, 8192, 8, 256, dtype="bf16", seed=0, seed_lo=4096, seed_hi=8192,
                             placement="runs")
    for row in inp.seed_idx:
        assert len(set(row.tolist())) == 256
        assert row.min() >= 4096 and row.max() < 8192
        runs = row.reshape(4, 64)
        for r in runs:
            assert np.array_equal(r, np.arange(r[0], r[0] + 64))


def test_score_inputs_spikes():
    s = W.make_score_inputs(200, 1000, 2, 5, seed=0, spike_frac=0.05)
    assert s.logits.shape == (200, 1000) and s.logits.dtype == np.uint16
    assert len(s.spiked_rows) == 10
    x = s.logits_f64()
    others = np.setdiff1d(np.arange(200), s.spiked_rows)
    assert (x[s.spiked_rows].max(axis=1) > 5.0).mean() >= 0.9
    assert (x[others].max(axis=1) > 7.5).sum() == 0


def test_named_workloads_shapes():
    w = W.WORKLOADS["gqa_l8192_stress"]
    assert (w.B, w.Hq, w.Hkv, w.L, w.D, w.S) == (4, 32, 8, 8192, 128, 256)
    assert abs(w.attn_flops - 4398.046511104e9) < 1e3
    assert W.WORKLOADS["llada_b8_l2048"].attn_flops == 4.0 * 8 * 32 * 2048 * 2048 * 128
