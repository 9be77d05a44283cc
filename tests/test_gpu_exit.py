"""Adaptive draft exit (Sec. 3.4, Eqs. 2-4) on the GPU, through the C ABI.

  * With the exit, greedy self-speculative output stays bit-identical to the
    GPU's own autoregressive output (the lossless property), for the paper's
    hyperparameters, a threshold near the drafts' typical confidence (so the
    exit point varies) and a threshold above 1 (one draft per round).
  * A zero threshold never exits: tokens and statistics equal the run without
    exit.
  * With an empty skip set every draft is accepted, AR_e = 1 > alpha in every
    round, and gamma falls by (1 - beta2) * eps per round: the final gamma has
    a closed form in the number of drafted rounds; the oracle's run ends at
    the same gamma.
  * With a static threshold, the draft counts of the GPU and of the oracle
    agree (confidence decisions are fp32 on the GPU, fp64 in the oracle, so
    only totals are compared).
"""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import common_prefix_runs, decoder

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

PAPER = (0.6, 0.9, 0.01, 0.5, 0.9)  # gamma0, alpha, eps, beta1, beta2


@pytest.fixture(scope="module")
def tiny_setup():
    w = synth.workloads()["tiny"]
    hw = synth.host_weights(w, seed=1)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    return w, hw, dw


def _typical_confidence(w, hw):
    orc = oracle.Oracle(w, hw, max_seq=160)
    prompt = synth.prompt(w.n_prompt, seed=0, vocab=w.vocab)
    _, _, dl, _ = orc.generate(prompt, 12, 8, mask=w.mask(), want_logits=True)
    return float(np.median([oracle.softmax_max(r) for r in dl]))


@pytest.mark.parametrize("K", [4, 8])
def test_exit_greedy_lossless(tiny_setup, K):
    w, hw, dw = tiny_setup
    dec = decoder(w, dw, 160)
    prompt = synth.prompt(w.n_prompt, seed=0, vocab=w.vocab)
    ar, _ = dec.generate(prompt, w.n_new, 0)
    g0 = _typical_confidence(w, hw)
    for params in (PAPER, (g0, 0.5, 0.0, 0.5, 1.0), (2.0, 0.9, 0.01, 0.5, 1.0)):
        dec.set_draft_exit(True, *params)
        sd, st = dec.generate(None, w.n_new, K)
        assert np.array_equal(ar, sd), params
        assert st["emitted"] == w.n_new == st["rounds"] + st["accepted"]
        assert st["drafted"] <= K * st["rounds"]
        if params[0] > 1.0:  # one draft in every round that drafts
            assert st["rounds"] - 1 <= st["drafted"] <= st["rounds"]
    dec.close()


def test_exit_zero_threshold_equals_no_exit(tiny_setup):
    w, hw, dw = tiny_setup
    dec = decoder(w, dw, 160)
    prompt = synth.prompt(w.n_prompt, seed=2, vocab=w.vocab)
    a, sa = dec.generate(prompt, w.n_new, w.K)
    dec.set_draft_exit(True, 0.0, 0.9, 0.01, 0.5, 1.0)
    b, sb = dec.generate(prompt, w.n_new, w.K)
    assert np.array_equal(a, b)
    for k in ("rounds", "drafted", "accepted", "emitted", "hist"):
        assert sa[k] == sb[k], k
    assert sb["gamma"] == 0.0
    dec.close()


def test_exit_empty_mask_gamma_closed_form(tiny_setup):
    w, hw, dw = tiny_setup
    zero = np.zeros(2 * w.n_layers, np.uint8)
    dec = decoder(w, dw, 160, mask=zero)
    dec.set_draft_exit(True, *PAPER)
    prompt = synth.prompt(w.n_prompt, seed=1, vocab=w.vocab)
    toks, st = dec.generate(prompt, w.n_new, w.K)
    assert st["accepted"] == st["drafted"]
    # the drafts' confidence (~1e-3 at these random weights) is below gamma,
    # so every drafting round stops after its first draft
    assert st["rounds"] - 1 <= st["drafted"] <= st["rounds"]
    assert st["gamma"] == pytest.approx(0.6 - 0.1 * 0.01 * st["drafted"], abs=2e-5)
    orc = oracle.Oracle(w, hw, max_seq=160)
    ref, rst = orc.generate(prompt, w.n_new, w.K, mask=zero, draft_exit=PAPER)
    assert np.array_equal(toks, ref)
    assert rst["drafted"] == st["drafted"] and rst["rounds"] == st["rounds"]
    assert rst["gamma"][-1] == pytest.approx(st["gamma"], abs=2e-5)
    dec.close()


@pytest.mark.parametrize("mode", [0, 1])
def test_exit_static_threshold_draft_counts_vs_oracle(tiny_setup, mode):
    """Draft counts of the GPU and of the oracle over the same tokens (the
    common prefix of their generations), with a static threshold near the
    drafts' typical confidence: the exit decisions are fp32 on the GPU and
    fp64 in the oracle, so the totals agree up to decisions at the threshold."""
    w, hw, dw = tiny_setup
    g0 = _typical_confidence(w, hw)
    params = (g0, 0.9, 0.0, 0.5, 1.0)
    dec = decoder(w, dw, 160)
    dec.set_sampling(1.0, 0.95)
    dec.set_draft_exit(True, *params)
    prompt = synth.prompt(w.n_prompt, seed=2, vocab=w.vocab)
    orc = oracle.Oracle(w, hw, max_seq=160)
    n, st, rst = common_prefix_runs(dec, orc, prompt, w.n_new, 8, mode=mode, seed=7, mask=w.mask(),
                                    top_p=0.95, draft_exit=params, min_common=16)
    assert st["emitted"] == n == st["rounds"] + st["accepted"]
    assert st["rounds"] - 1 <= st["drafted"] <= 8 * st["rounds"]
    assert abs(st["drafted"] - rst["drafted"]) <= max(4, rst["drafted"] // 8)
    dec.close()


def test_exit_bad_arguments(tiny_setup):
    import paper_2309_08168_gb300 as ssd
    w, hw, dw = tiny_setup
    dec = decoder(w, dw, 160)
    for bad in ((-0.1, 0.9, 0.01, 0.5, 0.9), (0.6, 1.5, 0.01, 0.5, 0.9), (0.6, 0.9, -0.01, 0.5, 0.9),
                (0.6, 0.9, 0.01, 1.5, 0.9), (0.6, 0.9, 0.01, 0.5, -0.1)):
        with pytest.raises(ssd.SSDError):
            dec.set_draft_exit(True, *bad)
    dec.set_draft_exit(False, -1.0, 2.0, -1.0, 3.0, 3.0)  # parameters are not checked when off
    prompt = synth.prompt(w.n_prompt, seed=0, vocab=w.vocab)
    a, st = dec.generate(prompt, 8, 4)
    assert st["gamma"] == 0.0
    dec.close()
