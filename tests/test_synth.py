"""Seeded input generator: rounding, distribution, determinism."""
import numpy as np
import torch

import synth


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(200000) * 0.02, rng.standard_normal(200000) * 37.0,
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.005859375, 3.0e-39])])
    ours = synth.round_bf16_host(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_weight_statistics_and_scale():
    a = synth.bf16_bits_to_f64(synth.fill_bf16_host(2_000_000, seed=3, tid=40))
    assert abs(a.mean()) < 1e-4
    assert abs(a.std() - 0.02) < 2e-4
    b = synth.bf16_bits_to_f64(synth.fill_bf16_host(2_000_000, seed=3, tid=40, scale=0.05))
    assert abs(b.std() - 0.001) < 2e-5
    # bounded support of Irwin-Hall(8): |z| <= 4.9 sigma
    assert np.max(np.abs(a)) < 0.02 * 4.9 * 1.01


def test_determinism_and_offsets():
    a = synth.fill_bf16_host(5000, seed=9, tid=3)
    b = synth.fill_bf16_host(5000, seed=9, tid=3)
    c = synth.fill_bf16_host(1000, seed=9, tid=3, first=2000)
    assert np.array_equal(a, b)
    assert np.array_equal(a[2000:3000], c)
    assert not np.array_equal(a, synth.fill_bf16_host(5000, seed=10, tid=3))
    assert not np.array_equal(a, synth.fill_bf16_host(5000, seed=9, tid=4))


def test_prompt_uniform():
    p = synth.prompt(64000, seed=1, vocab=32000)
    assert p.min() >= 0 and p.max() < 32000
    counts = np.bincount(p // 1000, minlength=32)
    assert counts.min() > 1700 and counts.max() < 2300


def test_skip_windows():
    w = synth.workloads()
    assert w["tiny"].skip == [2, 5]
    for name, L in (("llama2-7b", 32), ("llama2-13b", 40), ("llama2-70b", 80)):
        m = w[name].mask()
        assert m.sum() == L  # half of the 2L sublayers
        assert np.all(m[L // 2:(3 * L) // 2] == 1)


def test_algorithmic_bytes():
    w7 = synth.workloads()["llama2-7b"]
    full = synth.weight_bytes(w7)
    draft = synth.weight_bytes(w7, draft=True)
    assert abs(full / 1e9 - 13.215) < 0.01
    assert abs(draft / 1e9 - 6.739) < 0.01
