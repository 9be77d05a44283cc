"""Helpers shared by the GPU tests: decoders over synthetic workloads and the
tolerance rules of the parity contract."""
import numpy as np

import synth

ABS_TOL = 5e-2
REL_TOL = 1e-2
MARGIN = 0.1


def assert_logits_close(got, ref, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    excess = np.abs(got - ref) - (ABS_TOL + REL_TOL * np.abs(ref))
    i = np.unravel_index(np.argmax(excess), excess.shape)
    assert excess.max() <= 0, f"{what}: |gpu-oracle| exceeds tolerance at {i}: gpu {got[i]} oracle {ref[i]}"


def config_for(w, max_seq):
    import paper_2309_08168_gb300 as ssd
    return ssd.make_config(w.n_layers, w.d_model, w.n_heads, w.n_kv_heads, w.head_dim, w.ffn, w.vocab,
                           max_seq, w.rms_eps, w.rope_theta)


def decoder(w, weights_dev, max_seq, mask=None):
    import paper_2309_08168_gb300 as ssd
    dec = ssd.Decoder(config_for(w, max_seq), weights_dev, on_device=True)
    dec.set_skip(w.mask() if mask is None else mask)
    return dec


def check_tokens_vs_oracle(gpu_tokens, orc, prompt, n):
    """Greedy tokens must agree with the oracle's wherever the oracle's
    top-1 / top-2 margin exceeds 0.1; comparison stops at the first
    near-tie where they differ (the continuations then diverge).  Returns the
    number of positions compared."""
    ref, _ = orc.generate(prompt, n, 0)
    seq = np.concatenate([prompt, ref]).astype(np.int32)
    logits = orc.forward_uncached(seq[:-1])[len(prompt) - 1:]
    for i in range(n):
        top2 = np.sort(logits[i])[-2:]
        margin = top2[1] - top2[0]
        if gpu_tokens[i] != ref[i]:
            assert margin <= MARGIN, f"token {i}: gpu {gpu_tokens[i]} oracle {ref[i]} margin {margin}"
            return i
    return n


def common_prefix_runs(dec, orc, prompt, n_new, K, mode=0, seed=0, mask=None, top_p=1.0,
                       temperature=1.0, draft_exit=None, min_common=8):
    """Runs the GPU decoder and the oracle on the same generation and, where
    their tokens part (a near-tie decided in fp32 on one side and fp64 on the
    other), re-runs both with n_new cut to the common prefix, so that the
    statistics they return describe identical token sequences.  The decoder's
    skip set, sampling and draft-exit settings must already match the oracle
    arguments.  Returns (n, gpu stats, oracle stats) of the final runs;
    asserts that at least min_common tokens are shared."""
    n = n_new
    for _ in range(6):
        g, sg = dec.generate(prompt, n, K, mode=mode, seed=seed)
        o, so = orc.generate(prompt, n, K, mode=mode, seed=seed, temperature=temperature, top_p=top_p,
                             mask=mask, draft_exit=draft_exit)
        diff = np.nonzero(np.asarray(g) != np.asarray(o))[0]
        if diff.size == 0:
            assert n >= min_common, f"only {n} common tokens"
            return n, sg, so
        n = int(diff[0])
        assert n >= min_common, f"tokens part at {n}: gpu {g[n]} oracle {o[n]}"
    raise AssertionError("no common prefix found")
