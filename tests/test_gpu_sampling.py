"""Speculative sampling (Algorithm 4) on the GPU, checked by chi-square tests
against the target distribution:

  * the acceptance / resampling kernel in isolation on synthetic (p, q) over
    a 2048-token vocabulary, 500k rounds: the first emitted token follows p_0,
    and, given that j drafts were accepted, the next emitted token follows
    p_j;
  * end to end on the tiny config: the first token of a speculative round
    (drafted by the skip-set model, verified by the full model) follows the
    target's nucleus distribution computed by the fp64 oracle;
  * with an empty skip set every draft is accepted.
"""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import decoder

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
chi2 = pytest.importorskip("scipy.stats").chi2

P_MIN = 1e-3


def chi_square_p(counts, probs):
    n = counts.sum()
    exp = probs * n
    order = np.argsort(exp)
    # merge the smallest-expectation bins until every bin expects >= 5
    merged_c, merged_e, acc_c, acc_e = [], [], 0.0, 0.0
    for i in order:
        acc_c += counts[i]
        acc_e += exp[i]
        if acc_e >= 5:
            merged_c.append(acc_c)
            merged_e.append(acc_e)
            acc_c = acc_e = 0.0
    if acc_e > 0 and merged_e:
        merged_c[-1] += acc_c
        merged_e[-1] += acc_e
    c, e = np.array(merged_c), np.array(merged_e)
    stat = ((c - e) ** 2 / e).sum()
    return chi2.sf(stat, max(1, len(c) - 1))


@pytest.fixture(scope="module")
def tiny_dec():
    w = synth.workloads()["tiny"]
    hw = synth.host_weights(w, seed=1)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    dec = decoder(w, dw, 128)
    yield w, hw, dec
    dec.close()


def _dist(rng, V, alpha, zero_frac):
    p = rng.dirichlet(np.full(V, alpha))
    p[rng.random(V) < zero_frac] = 0.0
    return p / p.sum()


def test_accept_kernel_first_token_law(tiny_dec):
    w, hw, dec = tiny_dec
    rng = np.random.default_rng(0)
    V, T = w.vocab, 500_000
    p = np.stack([_dist(rng, V, 0.3, 0.2), _dist(rng, V, 0.3, 0.2)]).astype(np.float32)
    q = _dist(rng, V, 0.3, 0.2).astype(np.float32)[None, :]
    p64, q64 = p.astype(np.float64), q.astype(np.float64)
    drafts = rng.choice(V, size=(T, 1), p=q64[0] / q64[0].sum()).astype(np.int32)
    seeds = np.arange(T, dtype=np.uint64) * 7919 + 11
    n, y = dec.debug_spec_accept(p, q, drafts, seeds, pos0=100)
    assert set(np.unique(n)) <= {0, 1}
    first = np.where(n == 1, drafts[:, 0], y)
    counts = np.bincount(first, minlength=V).astype(np.float64)
    target = p64[0] / p64[0].sum()
    assert counts[target == 0].sum() == 0
    assert chi_square_p(counts, target) > P_MIN
    # acceptance rate = sum_x min(p, q)
    assert abs(n.mean() - np.minimum(p64[0], q64[0]).sum()) < 4e-3


def test_accept_kernel_later_positions(tiny_dec):
    w, hw, dec = tiny_dec
    rng = np.random.default_rng(1)
    V, Kd, T = w.vocab, 3, 400_000
    p = np.stack([_dist(rng, V, 0.5, 0.1) for _ in range(Kd + 1)]).astype(np.float32)
    q = np.stack([_dist(rng, V, 0.5, 0.1) for _ in range(Kd)]).astype(np.float32)
    qn = q.astype(np.float64) / q.astype(np.float64).sum(1, keepdims=True)
    drafts = np.stack([rng.choice(V, size=T, p=qn[j]) for j in range(Kd)], axis=1).astype(np.int32)
    seeds = np.arange(T, dtype=np.uint64) + 5
    n, y = dec.debug_spec_accept(p, q, drafts, seeds, pos0=7)
    for j in range(Kd + 1):
        reach = n >= j
        tok = np.where(n[reach] > j, drafts[reach, min(j, Kd - 1)], y[reach])
        counts = np.bincount(tok, minlength=V).astype(np.float64)
        target = p[j].astype(np.float64) / p[j].astype(np.float64).sum()
        assert chi_square_p(counts, target) > P_MIN, j


@pytest.mark.parametrize("temperature,top_p", [(0.1, 0.9), (1.0, 0.95)])
def test_end_to_end_first_token_law(tiny_dec, temperature, top_p):
    w, hw, dec = tiny_dec
    prompt = synth.prompt(w.n_prompt, seed=3, vocab=w.vocab)
    orc = oracle.Oracle(w, hw, max_seq=64)
    orc.prefill(prompt)
    logits = orc.forward(int(prompt[-1]), w.n_prompt - 1)
    target = oracle.nucleus_probs(logits, temperature, top_p)
    dec.set_sampling(temperature, top_p)
    dec.prefill(prompt)
    T = 12000
    first = np.empty(T, dtype=np.int64)
    acc = 0
    for s in range(T):
        toks, st = dec.generate(None, 2, 4, mode=1, seed=s)
        first[s] = toks[0]
        acc += st["accepted"]
    counts = np.bincount(first, minlength=w.vocab).astype(np.float64)
    # tokens outside the oracle's nucleus may only appear at its fp32 edge
    outside = counts[target == 0].sum()
    assert outside <= 0.002 * T
    keep = target > 0
    assert chi_square_p(counts[keep], target[keep] / target[keep].sum()) > P_MIN
    assert 0 < acc < T


def test_empty_mask_sampling_accepts_all(tiny_dec):
    w, hw, dec = tiny_dec
    dec.set_skip(np.zeros(2 * w.n_layers, np.uint8))
    dec.set_sampling(1.0, 0.95)
    prompt = synth.prompt(w.n_prompt, seed=0, vocab=w.vocab)
    toks, st = dec.generate(prompt, 40, 4, mode=1, seed=123)
    assert st["accepted"] == st["drafted"] > 0
    toks2, _ = dec.generate(None, 40, 4, mode=1, seed=123)
    assert np.array_equal(toks, toks2)  # deterministic for a seed
    dec.set_skip(w.mask())


# -- the LLaMA-2 vocabulary (V = 32000): each thread of the row kernels owns
# 32 tokens, and the nucleus threshold search runs over 32000 probabilities --

@pytest.fixture(scope="module")
def v32k_dec():
    w = synth.Workload("v32k", 2, 256, 4, 4, 64, 688, 32000, 32, 16, 4, 0, skip=[1, 2])
    hw = synth.host_weights(w, seed=2)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    dec = decoder(w, dw, 96)
    yield w, hw, dec
    dec.close()


def test_accept_kernel_first_token_law_v32k(v32k_dec):
    w, hw, dec = v32k_dec
    rng = np.random.default_rng(10)
    V, T = w.vocab, 500_000
    p = np.stack([_dist(rng, V, 0.3, 0.2), _dist(rng, V, 0.3, 0.2)]).astype(np.float32)
    q = _dist(rng, V, 0.3, 0.2).astype(np.float32)[None, :]
    p64, q64 = p.astype(np.float64), q.astype(np.float64)
    drafts = rng.choice(V, size=(T, 1), p=q64[0] / q64[0].sum()).astype(np.int32)
    seeds = np.arange(T, dtype=np.uint64) * 104729 + 3
    n, y = dec.debug_spec_accept(p, q, drafts, seeds, pos0=1000)
    first = np.where(n == 1, drafts[:, 0], y)
    counts = np.bincount(first, minlength=V).astype(np.float64)
    target = p64[0] / p64[0].sum()
    assert counts[target == 0].sum() == 0
    assert chi_square_p(counts, target) > P_MIN
    assert abs(n.mean() - np.minimum(p64[0], q64[0]).sum()) < 4e-3


def test_accept_kernel_later_positions_v32k(v32k_dec):
    w, hw, dec = v32k_dec
    rng = np.random.default_rng(11)
    V, Kd, T = w.vocab, 12, 300_000
    p = np.stack([_dist(rng, V, 0.5, 0.1) for _ in range(Kd + 1)]).astype(np.float32)
    # drafts close to the target so that later positions are reached often
    q = np.stack([0.7 * p[j].astype(np.float64) + 0.3 * _dist(rng, V, 0.5, 0.1) for j in range(Kd)])
    q = (q / q.sum(1, keepdims=True)).astype(np.float32)
    qn = q.astype(np.float64) / q.astype(np.float64).sum(1, keepdims=True)
    drafts = np.stack([rng.choice(V, size=T, p=qn[j]) for j in range(Kd)], axis=1).astype(np.int32)
    seeds = np.arange(T, dtype=np.uint64) + 77
    n, y = dec.debug_spec_accept(p, q, drafts, seeds, pos0=2000)
    for j in (0, 1, 2, 5):
        reach = n >= j
        assert reach.sum() > 20000, j
        tok = np.where(n[reach] > j, drafts[reach, min(j, Kd - 1)], y[reach])
        counts = np.bincount(tok, minlength=V).astype(np.float64)
        target = p[j].astype(np.float64) / p[j].astype(np.float64).sum()
        assert chi_square_p(counts, target) > P_MIN, j


@pytest.mark.parametrize("temperature,top_p", [(0.1, 0.9), (1.0, 0.95)])
def test_end_to_end_first_token_law_v32k(v32k_dec, temperature, top_p):
    """Nucleus (top-p) draft and target distributions over 32000 tokens: the
    first token of a speculative round follows the oracle's nucleus law."""
    w, hw, dec = v32k_dec
    prompt = synth.prompt(w.n_prompt, seed=4, vocab=w.vocab)
    orc = oracle.Oracle(w, hw, max_seq=64)
    orc.prefill(prompt)
    logits = orc.forward(int(prompt[-1]), w.n_prompt - 1)
    target = oracle.nucleus_probs(logits, temperature, top_p)
    dec.set_sampling(temperature, top_p)
    dec.prefill(prompt)
    T = 12000
    first = np.empty(T, dtype=np.int64)
    for s in range(T):
        toks, st = dec.generate(None, 2, 4, mode=1, seed=1000 + s)
        first[s] = toks[0]
    counts = np.bincount(first, minlength=w.vocab).astype(np.float64)
    outside = counts[target == 0].sum()
    assert outside <= 0.002 * T
    keep = target > 0
    # the nucleus holds at least top_p of the tempered mass and nothing below tau*
    assert keep.sum() < w.vocab or top_p == 1.0
    assert chi_square_p(counts[keep], target[keep] / target[keep].sum()) > P_MIN
