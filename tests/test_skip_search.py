"""Host logic of the skip-set search (Sec. 3.3): the local search over
single-bit flips of z, on objectives with known minima, and on a modelled
f(z) from the oracle's decoding (draft cost proportional to the sublayers it
runs, acceptance from the oracle's rounds)."""
import numpy as np
import pytest

import oracle
import synth
from paper_2309_08168_gb300 import skip_search as ss


def _separable(good, bad, L):
    def f(z):
        return 10.0 - sum(z[i] for i in good) + 2.0 * sum(z[i] for i in bad) + 0.1 * z.sum()
    return f


def test_finds_the_minimum_of_a_separable_objective():
    L = 12
    good, bad = [1, 4, 7, 10], [0, 2, 3, 5, 6, 8, 9, 11]
    f = ss.Objective(_separable(good, bad, L))
    z, v, hist = ss.local_search(f, np.zeros(L, np.uint8), budget=200, rng=np.random.default_rng(0))
    assert sorted(np.nonzero(z)[0].tolist()) == good
    assert v == pytest.approx(10.0 - 4 + 0.4)
    accepted = [h[1] for h in hist if h[2]]
    assert all(b < a for a, b in zip(accepted, accepted[1:]))  # every accepted step improves


def test_budget_max_skip_and_allowed_are_respected():
    L = 16
    f = ss.Objective(lambda z: -float(z.sum()))  # skipping everything is optimal
    z, v, _ = ss.local_search(f, np.zeros(L, np.uint8), budget=7, rng=np.random.default_rng(1))
    assert f.evals <= 7 and z.sum() <= 6
    f = ss.Objective(lambda z: -float(z.sum()))
    z, v, _ = ss.local_search(f, np.zeros(L, np.uint8), budget=100, rng=np.random.default_rng(2), max_skip=5)
    assert z.sum() == 5
    f = ss.Objective(lambda z: -float(z.sum()))
    z, v, _ = ss.local_search(f, np.zeros(L, np.uint8), budget=100, rng=np.random.default_rng(3),
                              allowed=[3, 9])
    assert np.nonzero(z)[0].tolist() == [3, 9]


def test_never_returns_worse_than_start_under_noise():
    rng = np.random.default_rng(5)
    L = 8
    base = _separable([2, 5], [0, 1, 3, 4, 6, 7], L)
    f = ss.Objective(lambda z: base(z) * (1.0 + 0.002 * rng.standard_normal()))
    start = np.zeros(L, np.uint8)
    z, v, _ = ss.local_search(f, start, budget=60, rng=np.random.default_rng(6))
    assert base(z) <= base(start)


def test_modelled_objective_on_the_oracle_prefers_the_scaled_skip_set(tiny, tiny_weights):
    """f(z) modelled from oracle runs: per round K draft steps costing the
    fraction of sublayers they run, plus one verification (cost 1); divided
    by the tokens emitted.  The tiny config scales the output projections of
    its skip set by 0.05, so skipping exactly those keeps acceptance high: the
    search started from the empty mask must end at least as good as it."""
    w, hw = tiny, tiny_weights
    L = 2 * w.n_layers
    prompt = synth.prompt(w.n_prompt, seed=0, vocab=w.vocab)
    orc = oracle.Oracle(w, hw, max_seq=w.max_seq())

    def modelled(z):
        _, st = orc.generate(prompt, 24, w.K, mask=z)
        run = 1.0 - z.sum() / L
        return (st["drafted"] * run + st["rounds"]) / st["emitted"]

    f = ss.Objective(modelled)
    z, v, _ = ss.local_search(f, np.zeros(L, np.uint8), budget=30, rng=np.random.default_rng(0))
    assert v <= f(w.mask()) + 1e-12
    assert v < f(np.zeros(L, np.uint8))
