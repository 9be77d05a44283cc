"""Pins for the oracle's forward pass (Sec. 3.2: p(x | z, x_1..x_i)).

The oracle is compared with things other than itself:
  * an independent torch fp64 composition of library ops (scaled dot-product
    attention, silu, complex-multiplication RoPE, repeat_interleave for GQA);
  * closed forms (RMSNorm of a constant vector, RoPE at position 0, RoPE's
    relative-position property, the all-sublayers-skipped model);
  * the brute-force full-sequence recomputation vs the cached incremental
    forward.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import synth
from conftest import micro_workload


def _t(bits):
    return torch.from_numpy(synth.bf16_bits_to_f64(np.asarray(bits)))


def torch_reference(w, weights, toks, n_full, mask):
    """Full-sequence forward from torch library ops, fp64.  Rows >= n_full
    run the masked model; they attend over the full model's keys/values for
    rows < n_full and their own for rows >= n_full (the draft reading)."""
    n = len(toks)
    d, H, Hkv, hd = w.d_model, w.n_heads, w.n_kv_heads, w.head_dim
    eps = w.rms_eps
    half = hd // 2
    h = _t(weights["embed"])[torch.as_tensor(np.asarray(toks, dtype=np.int64))].clone()
    pos = torch.arange(n, dtype=torch.float64)
    freq = w.rope_theta ** (-(2.0 * torch.arange(half, dtype=torch.float64)) / hd)
    rot = torch.polar(torch.ones(n, half, dtype=torch.float64), pos[:, None] * freq[None, :])

    def rms(x, g):
        return x * torch.rsqrt(x.pow(2).mean(-1, keepdim=True) + eps) * _t(g)

    def rope(x):  # x: [n, heads, hd]; pairs (i, i+half) as complex numbers
        z = torch.complex(x[..., :half], x[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    draft_rows = torch.arange(n) >= n_full
    for l, L in enumerate(weights["layers"]):
        skip_a = mask is not None and mask[2 * l]
        skip_m = mask is not None and mask[2 * l + 1]
        runs = ~draft_rows if skip_a else torch.ones(n, dtype=torch.bool)
        xn = rms(h, L["attn_norm"])
        q = rope((xn @ _t(L["wq"]).T).view(n, H, hd))
        k = rope((xn @ _t(L["wk"]).T).view(n, Hkv, hd))
        v = (xn @ _t(L["wv"]).T).view(n, Hkv, hd)
        k = k.repeat_interleave(H // Hkv, dim=1)
        v = v.repeat_interleave(H // Hkv, dim=1)
        allowed = torch.tril(torch.ones(n, n, dtype=torch.bool))
        allowed &= runs[None, :] | torch.eye(n, dtype=torch.bool)
        a = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           attn_mask=allowed)
        a = a.transpose(0, 1).reshape(n, H * hd)
        h = torch.where(runs[:, None], h + a @ _t(L["wo"]).T, h)
        runs_m = ~draft_rows if skip_m else torch.ones(n, dtype=torch.bool)
        xn = rms(h, L["mlp_norm"])
        mlp = (F.silu(xn @ _t(L["w_gate"]).T) * (xn @ _t(L["w_up"]).T)) @ _t(L["w_down"]).T
        h = torch.where(runs_m[:, None], h + mlp, h)
    return (rms(h, weights["final_norm"]) @ _t(weights["lm_head"]).T).numpy()


def _rel(a, b):
    return np.max(np.abs(a - b)) / max(1e-300, np.max(np.abs(b)))


@pytest.fixture(scope="module")
def micro():
    w = micro_workload()
    wts = synth.host_weights(w, seed=3)
    return w, wts


def test_uncached_matches_torch_full_model(micro):
    w, wts = micro
    toks = synth.prompt(9, seed=5, vocab=w.vocab)
    o = oracle.Oracle(w, wts, max_seq=32)
    got = o.forward_uncached(toks)
    ref = torch_reference(w, wts, toks, len(toks), None)
    assert _rel(got, ref) < 1e-10


def test_uncached_matches_torch_draft_rows(micro):
    w, wts = micro
    toks = synth.prompt(9, seed=6, vocab=w.vocab)
    mask = w.mask()
    assert mask.sum() == 2
    o = oracle.Oracle(w, wts, max_seq=32)
    got = o.forward_uncached(toks, n_full=5, mask=mask)
    ref = torch_reference(w, wts, toks, 5, mask)
    assert _rel(got, ref) < 1e-10


def test_tiny_matches_torch(tiny, tiny_weights):
    toks = synth.prompt(12, seed=2, vocab=tiny.vocab)
    o = oracle.Oracle(tiny, tiny_weights, max_seq=32)
    got = o.forward_uncached(toks, n_full=8, mask=tiny.mask())
    ref = torch_reference(tiny, tiny_weights, toks, 8, tiny.mask())
    assert _rel(got, ref) < 1e-10


def test_cached_equals_bruteforce(micro):
    """Incremental forward with KV cache (full rows, then draft rows that
    write and read the draft KV) == full recomputation."""
    w, wts = micro
    toks = synth.prompt(10, seed=7, vocab=w.vocab)
    mask = w.mask()
    o = oracle.Oracle(w, wts, max_seq=16)
    ref = o.forward_uncached(toks, n_full=6, mask=mask)
    for p in range(10):
        got = o.forward(int(toks[p]), p, mask=None if p < 6 else mask)
        assert _rel(got, ref[p]) < 1e-12, p


def test_cached_rewrite_after_draft(micro):
    """Draft rows write KV at positions the verification later rewrites: the
    full-model logits after the rewrite equal the all-full recomputation."""
    w, wts = micro
    toks = synth.prompt(8, seed=8, vocab=w.vocab)
    o = oracle.Oracle(w, wts, max_seq=16)
    for p in range(4):
        o.forward(int(toks[p]), p)
    for p in range(4, 8):  # drafts
        o.forward(int(toks[p]), p, mask=w.mask())
    ref = o.forward_uncached(toks)
    for p in range(4, 8):  # verification rewrites
        got = o.forward(int(toks[p]), p)
        assert _rel(got, ref[p]) < 1e-12


def test_all_skipped_closed_form(micro):
    """Every sublayer skipped: logits = W_head . RMSNorm(E[x])."""
    w, wts = micro
    o = oracle.Oracle(w, wts, max_seq=8)
    mask = np.ones(2 * w.n_layers, dtype=np.uint8)
    tok = 17
    got = o.forward(tok, 3, mask=mask)
    e = synth.bf16_bits_to_f64(wts["embed"][tok])
    xn = e / np.sqrt(np.mean(e * e) + w.rms_eps)
    ref = synth.bf16_bits_to_f64(wts["lm_head"]) @ xn
    assert _rel(got, ref) < 1e-12


def test_rmsnorm_constant_vector():
    d, c, eps = 64, 0.37, 1e-5
    g = synth.round_bf16_host(np.linspace(0.5, 1.5, d))
    out = oracle.rmsnorm(np.full(d, c), g, eps)
    ref = c / np.sqrt(c * c + eps) * synth.bf16_bits_to_f64(g)
    assert np.max(np.abs(out - ref)) < 1e-14


def test_rope_closed_forms():
    rng = np.random.default_rng(0)
    hd, theta = 8, 1e4
    x = rng.standard_normal(2 * hd)
    assert np.array_equal(oracle.rope(x, 2, hd, 0, theta), x)  # position 0: identity
    # explicit rotation of each pair (i, i+hd/2) by pos * theta^(-2i/hd)
    pos = 5
    got = oracle.rope(x[:hd], 1, hd, pos, theta)
    half = hd // 2
    for i in range(half):
        a = pos * theta ** (-2.0 * i / hd)
        assert abs(got[i] - (x[i] * np.cos(a) - x[i + half] * np.sin(a))) < 1e-14
        assert abs(got[i + half] - (x[i + half] * np.cos(a) + x[i] * np.sin(a))) < 1e-14
    # relative property: <R_m q, R_n k> = <R_{m-n} q, k>
    q, k = rng.standard_normal(hd), rng.standard_normal(hd)
    m, n = 37, 11
    lhs = oracle.rope(q, 1, hd, m, theta) @ oracle.rope(k, 1, hd, n, theta)
    rhs = oracle.rope(q, 1, hd, m - n, theta) @ k
    assert abs(lhs - rhs) < 1e-12


def test_rejects_bad_config(micro):
    w, wts = micro
    bad = micro_workload(n_kv_heads=3)
    with pytest.raises(ValueError):
        oracle.Oracle(bad, wts, max_seq=8)
