"""Skip-set search (Sec. 3.3) with the measured objective f(z) = GPU time of
the decoding loops per emitted token, on a LLaMA-2-7B-width model truncated to
4 layers (8 sublayers; skipping one saves ~100 MB of weight streaming per
draft step).  Started from the empty skip set, the search must find a skip
set that decodes faster per token, and the decoder keeps decoding correctly
with it (greedy output identical to its AR output)."""
import numpy as np
import pytest

import synth
from gpu_util import decoder

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def test_search_improves_on_the_empty_skip_set():
    from paper_2309_08168_gb300 import skip_search as ss
    w = synth.workloads()["llama2-7b"].truncated(4)
    dw = synth.device_weights(w, seed=0)
    torch.cuda.synchronize()
    L = 2 * w.n_layers
    dec = decoder(w, dw, 400, mask=np.zeros(L, np.uint8))
    prompts = [synth.prompt(64, seed=s, vocab=w.vocab) for s in range(2)]
    z, best, hist, f0 = ss.search_skip_set(dec, prompts, 48, 4, np.zeros(L, np.uint8), budget=14)
    assert 0 < z.sum() < L
    # re-measure both (timing noise): the found set must decode faster
    dec.set_skip(np.zeros(L, np.uint8))
    g0 = min(ss.ms_per_token(dec, prompts, 48, 4) for _ in range(2))
    dec.set_skip(z)
    g1 = min(ss.ms_per_token(dec, prompts, 48, 4) for _ in range(2))
    assert g1 < g0, (g0, g1, z)
    dec.prefill(prompts[0])
    ar, _ = dec.generate(None, 32, 0)
    sd, _ = dec.generate(None, 32, 4)
    assert np.array_equal(ar, sd)
    dec.close()
