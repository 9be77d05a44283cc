"""Pins for the oracle's adaptive draft exit (Sec. 3.4, Eqs. 2-4; Algorithms
3 / 4 of App. G).

  * The threshold recurrence (Eqs. 2-4) against closed forms: with a constant
    per-round acceptance AR_e the smoothed AR equals AR_e after the first
    update (beta1 = 0 there) and gamma moves by exactly (1 - beta2) * eps per
    round, up when AR <= alpha and down otherwise; beta2 = 1 freezes gamma;
    an alternating AR_e sequence gives the hand-derived smoothed values.
  * The confidence measure against hand-worked softmax maxima.
  * The exit rule at its extremes: gamma = 0 never exits (the run equals the
    one without exit, token for token and in its statistics); a gamma above
    1 exits after the first draft of every round.
  * With any threshold, greedy self-speculative decoding with exit still
    reproduces autoregressive decoding (the lossless property, Sec. 1).
  * With an empty skip set every draft is accepted, so each round's AR_e is
    1 > alpha and gamma falls by (1 - beta2) * eps per round: the final gamma
    has a closed form in the number of rounds.
  * In sampling mode the exit depends only on the draft distribution, so the
    first emitted token still follows the target's nucleus distribution p_0
    (chi-square over seeds, with a threshold that makes the exit point vary).
"""
import numpy as np
import pytest

import oracle
import synth
from conftest import micro_workload

PAPER = (0.6, 0.9, 0.01, 0.5, 0.9)  # gamma0, alpha, eps, beta1, beta2 (tab:Hyper, CNN/DM 13B)


def test_update_constant_low_acceptance_raises_gamma_linearly():
    st = (0.6, 0.0, 0)
    for e in range(1, 51):
        st = oracle.exit_update(st, PAPER, 0.5)
        assert st[1] == pytest.approx(0.5, abs=1e-15)
        assert st[0] == pytest.approx(0.6 + e * 0.1 * 0.01, abs=1e-12)
    assert st[2] == 50


def test_update_constant_high_acceptance_lowers_gamma_linearly():
    st = (0.6, 0.0, 0)
    for e in range(1, 31):
        st = oracle.exit_update(st, PAPER, 0.95)
        assert st[0] == pytest.approx(0.6 - e * 0.001, abs=1e-12)


def test_update_boundary_and_frozen_gamma():
    # AR == alpha counts as "AR <= alpha": gamma goes up
    st = oracle.exit_update((0.3, 0.0, 0), (0.3, 0.75, 0.02, 0.5, 0.5), 0.75)
    assert st[0] == pytest.approx(0.3 + 0.5 * 0.02, abs=1e-15)
    # beta2 = 1: gamma never moves
    st = (0.42, 0.0, 0)
    for a in (0.0, 1.0, 0.3, 0.99):
        st = oracle.exit_update(st, (0.42, 0.9, 0.05, 0.5, 1.0), a)
        assert st[0] == 0.42


def test_update_alternating_acceptance_hand_values():
    # AR_e = 1, 0, 1, 0, 1 with beta1 = 0.5 (beta1 = 0 at the first update)
    ar_expect = [1.0, 0.5, 0.75, 0.375, 0.6875]
    # alpha = 0.6: down, up, down, up, down by (1 - 0.9) * 0.01
    gamma_expect = [0.599, 0.6, 0.599, 0.6, 0.599]
    st = (0.6, 0.0, 0)
    for ar_e, a, g in zip([1, 0, 1, 0, 1], ar_expect, gamma_expect):
        st = oracle.exit_update(st, (0.6, 0.6, 0.01, 0.5, 0.9), ar_e)
        assert st[1] == pytest.approx(a, abs=1e-15)
        assert st[0] == pytest.approx(g, abs=1e-12)


def test_softmax_max_hand_cases():
    assert oracle.softmax_max(np.array([0.0, 0.0, np.log(2.0)])) == pytest.approx(0.5, abs=1e-15)
    assert oracle.softmax_max(np.zeros(7)) == pytest.approx(1.0 / 7.0, abs=1e-15)
    assert oracle.softmax_max(np.array([3.0, -40.0])) == pytest.approx(1.0 / (1.0 + np.exp(-43.0)), abs=1e-15)


@pytest.fixture(scope="module")
def micro():
    w = micro_workload()
    return w, synth.host_weights(w, seed=11)


def _gen(w, wts, K, n_new=24, mask=None, draft_exit=None, mode=0, seed=0, top_p=1.0):
    pr = synth.prompt(w.n_prompt, seed=4, vocab=w.vocab)
    o = oracle.Oracle(w, wts, max_seq=w.n_prompt + n_new + K + 1)
    return o.generate(pr, n_new, K, mode=mode, seed=seed, top_p=top_p,
                      mask=w.mask() if mask is None else mask, draft_exit=draft_exit)


@pytest.mark.parametrize("mode", [0, 1])
def test_zero_threshold_never_exits(micro, mode):
    w, wts = micro
    a, sa = _gen(w, wts, 4, mode=mode, seed=3, top_p=0.9)
    b, sb = _gen(w, wts, 4, mode=mode, seed=3, top_p=0.9, draft_exit=(0.0, 0.9, 0.01, 0.5, 1.0))
    assert np.array_equal(a, b)
    for k in ("rounds", "drafted", "accepted", "emitted", "hist"):
        assert sa[k] == sb[k]


@pytest.mark.parametrize("mode", [0, 1])
def test_threshold_above_one_drafts_once_per_round(micro, mode):
    w, wts = micro
    out, st = _gen(w, wts, 5, mode=mode, seed=5, top_p=0.9, draft_exit=(2.0, 0.9, 0.01, 0.5, 1.0))
    assert all(k == 1 for k in st["keff"][:-1])
    assert st["keff"][-1] in (0, 1)
    assert st["drafted"] == sum(st["keff"])
    assert st["emitted"] == 24 and st["emitted"] == st["rounds"] + st["accepted"]


def test_greedy_with_exit_is_lossless(micro):
    w, wts = micro
    ar, _ = _gen(w, wts, 0)
    # a threshold near the drafts' typical confidence makes the exit point vary
    _, _, dl, _ = oracle.Oracle(w, wts, max_seq=w.n_prompt + 40).generate(
        synth.prompt(w.n_prompt, seed=4, vocab=w.vocab), 8, 6, mask=w.mask(), want_logits=True)
    g0 = float(np.median([oracle.softmax_max(r) for r in dl]))
    for params in (PAPER, (g0, 0.5, 0.002, 0.5, 0.9), (g0, 0.9, 0.0, 0.5, 0.9)):
        ssd, st = _gen(w, wts, 6, draft_exit=params)
        assert np.array_equal(ar, ssd), params
        assert st["drafted"] == sum(st["keff"])
    _, st = _gen(w, wts, 6, draft_exit=(g0, 0.9, 0.0, 0.5, 0.9))
    assert len(set(st["keff"][:-1])) > 1  # the exit point does vary


def test_empty_mask_gamma_closed_form(micro):
    w, wts = micro
    zero = np.zeros(2 * w.n_layers, dtype=np.uint8)
    # every draft is accepted: AR_e = 1 > alpha in every round with drafts
    out, st = _gen(w, wts, 4, mask=zero, draft_exit=PAPER)
    assert st["accepted"] == st["drafted"]
    g = 0.6
    for k, got in zip(st["keff"], st["gamma"]):
        if k > 0:
            g -= 0.1 * 0.01
        assert got == pytest.approx(g, abs=1e-12)


def test_sampling_with_exit_keeps_the_first_token_law():
    """The exit decision depends only on the draft distribution q, so the
    speculative-sampling guarantee is untouched: the first emitted token
    still follows the target's nucleus distribution p_0 (Alg. 4)."""
    from scipy.stats import chi2
    w = micro_workload(vocab=16, n_prompt=3)
    wts = synth.host_weights(w, seed=21)
    pr = synth.prompt(3, seed=2, vocab=w.vocab)
    o = oracle.Oracle(w, wts, max_seq=12)
    o.prefill(pr)
    p0 = oracle.nucleus_probs(o.forward(int(pr[-1]), 2) * 40.0, 1.0, 0.95)
    T = 2500
    toks = np.empty(T, dtype=np.int64)
    keff = np.empty(T, dtype=np.int64)
    for s in range(T):
        out, st = o.generate(pr, 5, 3, mode=1, seed=5000 + s, temperature=1 / 40, top_p=0.95, mask=w.mask(),
                             draft_exit=(0.8, 0.9, 0.0, 0.5, 1.0))
        toks[s] = out[0]
        keff[s] = st["keff"][0]
    assert len(set(keff.tolist())) > 1  # the first round's exit point varies with the draws
    counts = np.bincount(toks, minlength=w.vocab)
    keep = p0 * T >= 5
    assert counts[~keep].sum() <= max(10, 3 * p0[~keep].sum() * T)
    exp = p0[keep] * T
    stat = ((counts[keep] - exp) ** 2 / exp).sum() + 0.0
    assert chi2.sf(stat, max(1, keep.sum() - 1)) > 1e-4, (counts, p0 * T)
