"""Bounded device waits: a grid barrier of the forward kernel that can never
complete gives up after its wait limit, the call returns SSD_ERR_TIMEOUT and
the handle keeps working.

The failure is made on purpose without faulting anything: a test hook of the
library raises the target of one grid barrier by one arrival (no CTA will
ever bring it), with a wait limit of 50 ms.  Every CTA then records the
timeout, lets its copies in flight land and returns; the host reads the
status.  The next forward, without the hook, must give the same logits, bit
for bit, as the same forward before the failure.
"""
import numpy as np
import pytest

import synth
from gpu_util import decoder

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.mark.parametrize("barrier", [1, 3, 5])
def test_unreachable_barrier_times_out_and_handle_recovers(barrier):
    import paper_2309_08168_gb300 as ssd
    w = synth.workloads()["tiny"]
    hw = synth.host_weights(w, seed=1)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    dec = decoder(w, dw, 128)
    prompt = synth.prompt(w.n_prompt, seed=3, vocab=w.vocab)
    rows = synth.prompt(5, seed=4, vocab=w.vocab)
    dec.prefill(prompt)
    before = dec.debug_forward(False, rows, w.n_prompt - 1)

    dec.debug_stall_barrier(barrier, 0.05)
    with pytest.raises(ssd.SSDError) as e:
        dec.debug_forward(False, rows, w.n_prompt - 1)
    assert e.value.code == ssd.SSD_ERR_TIMEOUT
    assert "timed out" in str(e.value)

    after = dec.debug_forward(False, rows, w.n_prompt - 1)
    assert np.array_equal(before.view(np.uint32), after.view(np.uint32))
    ar, _ = dec.generate(prompt, 16, 0)
    sd, _ = dec.generate(None, 16, 4)
    assert np.array_equal(ar, sd)
    dec.close()


def test_stall_hook_arguments():
    import paper_2309_08168_gb300 as ssd
    w = synth.workloads()["tiny"]
    hw = synth.host_weights(w, seed=1)
    dw = synth.host_to_device_weights(hw)
    dec = decoder(w, dw, 64)
    for bad in ((-1, 0.05), (1, 0.0), (1, 11.0)):
        with pytest.raises(ssd.SSDError) as e:
            dec.debug_stall_barrier(*bad)
        assert e.value.code == ssd.SSD_ERR_INVALID_ARG
    dec.debug_stall_barrier(0, 1.0)  # disarmed: the next forward runs normally
    dec.prefill(synth.prompt(8, seed=0, vocab=w.vocab))
    dec.debug_forward(False, synth.prompt(2, seed=1, vocab=w.vocab), 7)
    dec.close()
