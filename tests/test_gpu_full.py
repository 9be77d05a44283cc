"""Full-size LLaMA-2-7B-shaped workload (32 layers, d 4096, vocab 32000,
prompt 512, 512 new tokens, K = 8, skip set = the 32 middle sublayers), in the
launch configuration bench.py times:

  * greedy self-speculative output == the GPU's own plain AR output, bit for
    bit, over all 512 tokens (a property that holds at any size);
  * sampled outputs the oracle can compute one by one: verification and
    draft logits of the full-depth 7B model after a 16-token prompt, against
    the fp64 oracle on the same bf16 weights.
"""
import os

import numpy as np
import pytest

import oracle
import synth
from gpu_util import assert_logits_close, decoder

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def _mem_available_gb():
    try:
        for line in open("/proc/meminfo"):
            if line.startswith("MemAvailable"):
                return int(line.split()[1]) / 1e6
    except OSError:
        pass
    return 0.0


@pytest.fixture(scope="module")
def w7():
    return synth.workloads()["llama2-7b"]


@pytest.fixture(scope="module")
def dev7(w7):
    dw = synth.device_weights(w7, seed=0)
    torch.cuda.synchronize()
    yield dw
    del dw
    torch.cuda.empty_cache()


def test_7b_greedy_ssd_bit_identical_to_ar(w7, dev7):
    dec = decoder(w7, dev7, w7.max_seq())
    prompt = synth.prompt(w7.n_prompt, seed=0, vocab=w7.vocab)
    ar, st_ar = dec.generate(prompt, w7.n_new, 0)
    sd, st = dec.generate(None, w7.n_new, w7.K)
    assert np.array_equal(ar, sd)
    assert st["emitted"] == w7.n_new and st["drafted"] > 0
    print(f"\n7B: accept rate {st['accept_rate']:.3f}, tokens/round {w7.n_new / st['rounds']:.2f}, "
          f"AR {st_ar['total_ms']:.1f} ms, SSD {st['total_ms']:.1f} ms")
    dec.close()


@pytest.mark.skipif(_mem_available_gb() < 40, reason="needs ~16 GB of host memory for the fp64 oracle")
def test_7b_sampled_logits_vs_oracle(w7, dev7):
    hw = synth.host_weights(w7, seed=0)
    orc = oracle.Oracle(w7, hw, max_seq=64)
    dec = decoder(w7, dev7, 64)
    prompt = synth.prompt(16, seed=5, vocab=w7.vocab)
    rows = np.concatenate([prompt[-1:], synth.prompt(w7.K, seed=6, vocab=w7.vocab)])
    dec.prefill(prompt)
    got = dec.debug_forward(False, rows, 15)
    orc.prefill(prompt)
    for r in range(len(rows)):
        ref = orc.forward(int(rows[r]), 15 + r)
        assert_logits_close(got[r], ref, f"7B verify row {r}")
    # draft step 1 (skip-set model) at position 15
    got_d = dec.debug_forward(True, rows[:1], 15)
    orc2 = oracle.Oracle(w7, hw, max_seq=64)
    orc2.prefill(prompt)
    ref_d = orc2.forward(int(rows[0]), 15, mask=w7.mask())
    assert_logits_close(got_d[0], ref_d, "7B draft")
    dec.close()
