"""Oracle parity of the verification and draft forwards at contexts that span
several attention segments.

The forward kernel splits attention over absolute 128-position segments and
combines each KV head's segment partials in segment order; every context of
the benchmark workloads (512-2061 positions) goes through that combine.  Here
the GPU logits are compared with the fp64 oracle, element by element at
|d| <= 5e-2 + 1e-2 |oracle|, after prompts of 125-400 tokens:

  * tiny (4 layers, d 256): 300-token prompt, verification over 1, 5, 9, 13
    and 16 rows (every input-plane class) and the draft rows one by one;
    rows straddling the segment boundaries at 128 and 256; a 2070-token
    prompt, past the 16 segments the combine folds in one batch;
  * LLaMA-2-7B widths (2 layers, 32 heads): 400-token prompt, 9 rows;
  * LLaMA-2-70B widths (2 layers, GQA 64 query / 8 KV heads): 300-token
    prompt, 9 rows, so 72 query vectors of each KV head meet several
    segments;
  * LLaMA-2-13B widths (2 layers, d 5120, FFN 13824): 200-token prompt, 13
    rows (the 13B sampling workload's K + 1), and a 16-token prompt;
  * batch invariance across segment boundaries: every row of a 16-row
    forward straddling position 256 equals, bit for bit, the one-row forward.

The sequence is the decoding loop's: prefill, then the draft rows one at a
time (the skip-set model writes KV only in the attention sublayers it runs),
then one verification forward over all rows (Algorithm 2's verification
stage attends over the committed cache plus the drafts).  The oracle runs the
same sequence with its cached fp64 forward.
"""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import assert_logits_close, decoder

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def draft_then_verify(w, hw, dw, P, n_rows, seed, max_seq, mask=None):
    """GPU and oracle logits of n_rows draft steps, then of one verification
    forward over the same rows, at positions P-1 .. P-2+n_rows after a
    P-token prompt.  Returns (gpu draft, oracle draft, gpu verify, oracle
    verify), each [n_rows][vocab]."""
    mask = w.mask() if mask is None else mask
    prompt = synth.prompt(P, seed=seed, vocab=w.vocab)
    rows = np.concatenate([prompt[-1:], synth.prompt(n_rows - 1, seed=seed + 1, vocab=w.vocab)]) \
        if n_rows > 1 else prompt[-1:]
    dec = decoder(w, dw, max_seq, mask=mask)
    dec.prefill(prompt)
    got_d = np.stack([dec.debug_forward(True, rows[j:j + 1], P - 1 + j)[0] for j in range(n_rows)])
    got_v = dec.debug_forward(False, rows, P - 1)
    dec.close()
    orc = oracle.Oracle(w, hw, max_seq=max_seq)
    orc.prefill(prompt)
    ref_d = np.stack([orc.forward(int(rows[j]), P - 1 + j, mask=mask) for j in range(n_rows)])
    ref_v = np.stack([orc.forward(int(rows[r]), P - 1 + r) for r in range(n_rows)])
    orc.close()
    return got_d, ref_d, got_v, ref_v


@pytest.fixture(scope="module")
def tiny_setup():
    w = synth.workloads()["tiny"]
    hw = synth.host_weights(w, seed=1)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    return w, hw, dw


@pytest.mark.parametrize("n_rows", [1, 5, 9, 13, 16])
def test_tiny_three_segments(tiny_setup, n_rows):
    w, hw, dw = tiny_setup
    got_d, ref_d, got_v, ref_v = draft_then_verify(w, hw, dw, 300, n_rows, seed=21, max_seq=320)
    assert_logits_close(got_v, ref_v, f"tiny verify M={n_rows} at 299")
    assert_logits_close(got_d, ref_d, f"tiny draft rows at 299")


def test_tiny_beyond_one_combine_batch(tiny_setup):
    """Contexts past 16 segments (2048 positions): the combine folds a second
    batch of segment partials into running sums rescaled to the new maximum.
    A 2070-token prompt (two prefill chunks), 9 verification rows and the
    draft rows at positions 2069 .. 2077 (17 segments)."""
    w, hw, dw = tiny_setup
    got_d, ref_d, got_v, ref_v = draft_then_verify(w, hw, dw, 2070, 9, seed=51, max_seq=2100)
    assert_logits_close(got_v, ref_v, "tiny verify M=9 at 2069")
    assert_logits_close(got_d, ref_d, "tiny draft rows at 2069")


@pytest.mark.parametrize("P", [125, 253])
def test_tiny_rows_straddle_segment_boundary(tiny_setup, P):
    """Rows P-1 .. P+7 cross the segment boundary at 128 (P = 125) or 256
    (P = 253): rows of one forward see different numbers of segments."""
    w, hw, dw = tiny_setup
    got_d, ref_d, got_v, ref_v = draft_then_verify(w, hw, dw, P, 9, seed=31, max_seq=288)
    assert_logits_close(got_v, ref_v, f"tiny verify straddling, P={P}")
    assert_logits_close(got_d, ref_d, f"tiny draft straddling, P={P}")


def test_batch_invariance_across_segments(tiny_setup):
    w, hw, dw = tiny_setup
    dec = decoder(w, dw, 300)
    dec.prefill(synth.prompt(249, seed=5, vocab=w.vocab))
    rows = synth.prompt(16, seed=6, vocab=w.vocab)
    many = dec.debug_forward(False, rows, 248)  # positions 248 .. 263
    one = np.stack([dec.debug_forward(False, rows[r:r + 1], 248 + r)[0] for r in range(16)])
    assert np.array_equal(many.view(np.uint32), one.view(np.uint32))
    dec.close()


def _big(shape, n_layers=2, seed=7):
    w = synth.workloads()[shape].truncated(n_layers)
    hw = synth.host_weights(w, seed=seed)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    return w, hw, dw


@pytest.mark.parametrize("shape,P,n_rows", [("llama2-7b", 400, 9), ("llama2-70b", 300, 9),
                                            ("llama2-13b", 200, 13), ("llama2-13b", 16, 9)])
def test_big_widths_long_context(shape, P, n_rows):
    w, hw, dw = _big(shape)
    got_d, ref_d, got_v, ref_v = draft_then_verify(w, hw, dw, P, n_rows, seed=41, max_seq=P + 32)
    assert_logits_close(got_v, ref_v, f"{shape} verify M={n_rows} at {P - 1}")
    assert_logits_close(got_d[:3], ref_d[:3], f"{shape} draft at {P - 1}")
    del dw
    torch.cuda.empty_cache()


def test_13b_widths_ssd_equals_ar():
    """The 13B sampling workload's K = 12 (13-row verification) at 13B widths:
    greedy self-speculative output bit-identical to the GPU's AR output."""
    w, hw, dw = _big("llama2-13b")
    dec = decoder(w, dw, 200)
    prompt = synth.prompt(100, seed=3, vocab=w.vocab)
    ar, _ = dec.generate(prompt, 64, 0)
    sd, st = dec.generate(None, 64, 12)
    assert np.array_equal(ar, sd)
    assert st["emitted"] == 64
    dec.close()
