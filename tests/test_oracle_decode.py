"""Pins for the oracle's decoding loops and sampling arithmetic.

  * Philox4x32-10 against the published known-answer vectors.
  * Nucleus / temperature / inverse-CDF draws against hand-worked cases.
  * Greedy self-speculative decoding (Algorithm 2) reproduces greedy
    autoregressive decoding (Algorithm 1) token for token: the paper's
    lossless property (Sec. 1, App. G.2), for several masks and K.
  * With an empty skip set the draft model is the original model
    (Algorithm 2's definition of p(x|0, ...)), so every draft is accepted, in
    greedy and in sampling mode.
  * Speculative sampling (Algorithm 4): the exact output law of one
    verification step, integrated over its uniforms on a grid, equals p; a
    Monte Carlo run checks the law of later positions.
"""
import json
import os

import numpy as np
import pytest

import oracle
import synth
from conftest import micro_workload

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_philox_known_answers():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt"))
            if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = oracle.philox(v[0:4], v[4:6])
        assert [int(x) for x in out] == v[6:10]


def test_uniform_open_interval_and_counter():
    us = [oracle.uniform(123, p, k) for p in range(200) for k in range(3)]
    assert all(0.0 < u < 1.0 for u in us)
    assert len(set(us)) == len(us)
    # counter (0,0,0,0) with key 0: first word of the first known answer
    assert oracle.uniform(0, 0, 0) == (0x6627E8D5 + 0.5) / 2 ** 32


def test_nucleus_golden():
    cases = json.load(open(os.path.join(GOLDEN, "sampling_cases.json")))
    for c in cases["nucleus"]:
        logits = np.array(c["logits"]) if "logits" in c else np.log(np.array(c["probs"]))
        got = oracle.nucleus_probs(logits, c["temperature"], c["top_p"])
        np.testing.assert_allclose(got, c["expect"], atol=1e-12)


def test_sample_golden():
    cases = json.load(open(os.path.join(GOLDEN, "sampling_cases.json")))
    for c in cases["sample"]:
        assert oracle.sample(np.array(c["probs"]), c["u"]) == c["expect"], c


def test_argmax_lowest_index_on_ties():
    assert oracle.argmax(np.array([1.0, 3.0, 3.0, 2.0])) == 1
    assert oracle.argmax(np.array([5.0])) == 0


@pytest.fixture(scope="module")
def micro():
    w = micro_workload()
    return w, synth.host_weights(w, seed=11)


def _run(w, wts, K, mask, n_new=20, mode=0, seed=0, temperature=1.0, top_p=1.0, prompt_seed=4):
    pr = synth.prompt(w.n_prompt, seed=prompt_seed, vocab=w.vocab)
    o = oracle.Oracle(w, wts, max_seq=w.n_prompt + n_new + K + 1)
    return o.generate(pr, n_new, K, mode=mode, seed=seed, temperature=temperature, top_p=top_p, mask=mask)


@pytest.mark.parametrize("K", [1, 2, 3, 5])
@pytest.mark.parametrize("mask_kind", ["default", "all", "random"])
def test_greedy_ssd_equals_ar(micro, K, mask_kind):
    w, wts = micro
    if mask_kind == "default":
        mask = w.mask()
    elif mask_kind == "all":
        mask = np.ones(2 * w.n_layers, dtype=np.uint8)
    else:
        mask = np.random.default_rng(K).integers(0, 2, 2 * w.n_layers).astype(np.uint8)
    ar, st_ar = _run(w, wts, 0, None)
    ssd, st = _run(w, wts, K, mask)
    assert np.array_equal(ar, ssd)
    assert st["emitted"] == 20 and st_ar["rounds"] == 20
    assert st["rounds"] == sum(st["hist"])
    assert st["emitted"] == st["rounds"] + st["accepted"]


def test_greedy_ssd_equals_ar_tiny(tiny, tiny_weights):
    pr = synth.prompt(tiny.n_prompt, seed=0, vocab=tiny.vocab)
    o = oracle.Oracle(tiny, tiny_weights, max_seq=tiny.max_seq())
    ar, _ = o.generate(pr, 24, 0)
    ssd, st = o.generate(pr, 24, tiny.K, mask=tiny.mask())
    assert np.array_equal(ar, ssd)
    assert st["accepted"] > 0  # the 0.05-scaled skip set makes drafts useful


def test_empty_mask_accepts_everything(micro):
    w, wts = micro
    zero = np.zeros(2 * w.n_layers, dtype=np.uint8)
    for mode in (0, 1):
        out, st = _run(w, wts, 4, zero, n_new=21, mode=mode, seed=9, top_p=0.9)
        assert st["accepted"] == st["drafted"]
        # every round but the last drafts K=4 and emits K+1
        assert st["hist"][4] == st["rounds"] - 1


def test_edge_lengths(micro):
    w, wts = micro
    for n_new in (0, 1, 2):
        out, st = _run(w, wts, 3, w.mask(), n_new=n_new)
        assert st["emitted"] == n_new
        ar, _ = _run(w, wts, 0, None, n_new=n_new)
        assert np.array_equal(out, ar)
    # prompt of one token: no prefill forward at all
    o = oracle.Oracle(w, wts, max_seq=16)
    a, _ = o.generate(np.array([5], dtype=np.int32), 6, 0)
    b, _ = o.generate(np.array([5], dtype=np.int32), 6, 3, mask=w.mask())
    assert np.array_equal(a, b)


def test_capacity_and_bad_args(micro):
    w, wts = micro
    o = oracle.Oracle(w, wts, max_seq=10)
    pr = synth.prompt(6, seed=1, vocab=w.vocab)
    with pytest.raises(ValueError):
        o.generate(pr, 5, 3)  # 6 + 5 + 3 + 1 > 10
    with pytest.raises(ValueError):
        o.generate(pr, 1, 0, mode=1, temperature=0.0)


def _law_grid(p, q, G):
    """Exact output law of the first emitted token of a one-draft round,
    integrated over d ~ q and the two uniforms on a G x G midpoint grid."""
    V = p.shape[1]
    mids = (np.arange(G) + 0.5) / G
    d = np.repeat(np.arange(V), G * G)
    r = np.tile(np.repeat(mids, G), V)
    u = np.tile(mids, V * G)
    ures = np.stack([u, u], axis=1)
    n, y = oracle.spec_verify_batch(p, q[None, :], d[:, None], r[:, None], ures)
    first = np.where(n == 1, d, y)
    weights = q[d] / (G * G)
    return np.bincount(first, weights=weights, minlength=V)


def test_spec_verify_exact_law():
    rng = np.random.default_rng(1)
    V = 6
    for trial in range(4):
        p0 = rng.random(V) ** 2
        p0[rng.integers(V)] = 0.0
        p0 /= p0.sum()
        q = rng.random(V) ** 2
        q[rng.integers(V)] = 0.0
        q /= q.sum()
        p = np.stack([p0, rng.dirichlet(np.ones(V))])
        law = _law_grid(p, q, 400)
        assert np.max(np.abs(law - p0)) < 6e-3, (law, p0)


def test_spec_verify_later_positions_monte_carlo():
    """Kd = 3 with fixed target rows: conditional on reaching position j, the
    emitted token there follows p_{j-1} (chi-square, Monte Carlo)."""
    from scipy.stats import chi2
    rng = np.random.default_rng(2)
    V, Kd, T = 8, 3, 400000
    p = rng.dirichlet(np.ones(V), size=Kd + 1)
    q = rng.dirichlet(np.ones(V), size=Kd)
    drafts = np.stack([rng.choice(V, size=T, p=q[j]) for j in range(Kd)], axis=1)
    r = rng.random((T, Kd))
    ures = rng.random((T, Kd + 1))
    n, y = oracle.spec_verify_batch(p, q, drafts, r, ures)
    for j in range(Kd + 1):  # emitted index j (0-based) exists iff n >= j
        reach = n >= j
        tok = np.where(n[reach] > j, drafts[reach, min(j, Kd - 1)], y[reach])
        counts = np.bincount(tok, minlength=V)
        exp = p[j] * reach.sum()
        stat = ((counts - exp) ** 2 / exp).sum()
        assert chi2.sf(stat, V - 1) > 1e-4, (j, counts, exp)


def test_sampling_generate_first_token_law():
    """End to end through orc_generate (drafts from the masked model, target
    from the full model): the first emitted token of a one-draft round
    follows the target's nucleus distribution p_0."""
    from scipy.stats import chi2
    w = micro_workload(vocab=16, n_prompt=3)
    wts = synth.host_weights(w, seed=21)
    pr = synth.prompt(3, seed=2, vocab=w.vocab)
    o = oracle.Oracle(w, wts, max_seq=8)
    o.prefill(pr)
    logits = o.forward(int(pr[-1]), 2)
    p0 = oracle.nucleus_probs(logits * 40.0, 1.0, 0.95)  # sharpen: non-trivial nucleus
    T = 3000
    toks = np.empty(T, dtype=np.int64)
    acc = 0
    # scale logits through temperature instead: temperature 1/40
    for s in range(T):
        out, st = o.generate(pr, 2, 2, mode=1, seed=1000 + s, temperature=1 / 40, top_p=0.95, mask=w.mask())
        toks[s] = out[0]
        acc += st["accepted"]
    counts = np.bincount(toks, minlength=w.vocab)
    keep = p0 * T >= 5
    assert counts[~keep].sum() <= max(10, 3 * p0[~keep].sum() * T)
    exp = p0[keep] * T
    stat = ((counts[keep] - exp) ** 2 / exp).sum() + 0.0
    assert chi2.sf(stat, max(1, keep.sum() - 1)) > 1e-4, (counts, p0 * T)
    assert 0 < acc < T  # both branches (accept and resample) exercised
