"""The tensor-core prefill (prompt encoding, Sec. 3.1) against the fp64 oracle.

Prompts longer than 16 tokens are encoded by the prefill kernels: tcgen05
GEMMs for every projection and a causal flash-attention kernel, chunk by
chunk of up to 2048 positions.  Its result is the KV cache of the prompt,
which every later forward reads, so it is checked through the logits of the
last prompt row (the first decoding round's x_last, computed by the decode
kernel over the prefilled cache), element by element against the oracle at
|d| <= 5e-2 + 1e-2 |oracle|:

  * 2 layers at LLaMA-2-7B widths after 512 prompt tokens (the 7B workload's
    prompt), plus greedy self-speculative output == AR output after it;
  * 2 layers at LLaMA-2-13B widths after 1536 prompt tokens (the 13B
    sampling workload's prompt);
  * the tiny model after 2100 prompt tokens: two prefill chunks, attention
    over more than 2048 keys;
  * prompt lengths around the 128-row tile of the GEMMs and the 64-row
    blocks of the attention kernel (17, 127, 129, 200 tokens).
"""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import assert_logits_close, decoder

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def last_row_logits(w, hw, dw, P, seed, max_seq, extra_rows=0):
    """GPU and oracle logits of the rows [prompt[-1], extra...] at positions
    P-1.. after prefilling a P-token prompt."""
    prompt = synth.prompt(P, seed=seed, vocab=w.vocab)
    rows = np.concatenate([prompt[-1:], synth.prompt(extra_rows, seed=seed + 1, vocab=w.vocab)]) \
        if extra_rows else prompt[-1:]
    dec = decoder(w, dw, max_seq)
    dec.prefill(prompt)
    got = dec.debug_forward(False, rows, P - 1)
    orc = oracle.Oracle(w, hw, max_seq=max_seq)
    orc.prefill(prompt)
    ref = np.stack([orc.forward(int(rows[r]), P - 1 + r) for r in range(len(rows))])
    orc.close()
    return dec, prompt, got, ref


def test_7b_widths_prompt_512():
    w = synth.workloads()["llama2-7b"].truncated(2)
    hw = synth.host_weights(w, seed=9)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    dec, prompt, got, ref = last_row_logits(w, hw, dw, 512, seed=51, max_seq=600, extra_rows=8)
    assert_logits_close(got, ref, "7B widths after a 512-token prefill")
    ar, _ = dec.generate(prompt, 48, 0)
    sd, st = dec.generate(None, 48, 8)
    assert np.array_equal(ar, sd)
    dec.close()


def test_13b_widths_prompt_1536():
    w = synth.workloads()["llama2-13b"].truncated(2)
    hw = synth.host_weights(w, seed=10)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    dec, prompt, got, ref = last_row_logits(w, hw, dw, 1536, seed=52, max_seq=1560)
    assert_logits_close(got, ref, "13B widths after a 1536-token prefill")
    dec.close()


@pytest.fixture(scope="module")
def tiny_setup():
    w = synth.workloads()["tiny"]
    hw = synth.host_weights(w, seed=1)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    return w, hw, dw


def test_tiny_two_chunks(tiny_setup):
    w, hw, dw = tiny_setup
    dec, prompt, got, ref = last_row_logits(w, hw, dw, 2100, seed=53, max_seq=2200, extra_rows=4)
    assert_logits_close(got, ref, "tiny after a 2100-token prefill (two chunks)")
    ar, _ = dec.generate(prompt, 32, 0)
    sd, _ = dec.generate(None, 32, 4)
    assert np.array_equal(ar, sd)
    dec.close()


@pytest.mark.parametrize("P", [17, 127, 129, 200])
def test_tiny_tile_edges(tiny_setup, P):
    w, hw, dw = tiny_setup
    dec, prompt, got, ref = last_row_logits(w, hw, dw, P, seed=54 + P, max_seq=256, extra_rows=3)
    assert_logits_close(got, ref, f"tiny after a {P}-token prefill")
    dec.close()
