"""ssd_linear_noalloc, the allocation-free projection, through the C ABI.

It serves callers that cannot allocate device memory when they need a
projection (all of HBM reserved up front, allocations owned by a host
framework, or a loop that must not risk the device-wide synchronisation of
cudaMalloc / cudaFree): it runs the decoder's projection GEMM with its split-K
scratch in fixed device arrays of the library.  Its output must match what
the existing entry point produces with the same kernel: the logits of
ssd_debug_forward when every sublayer is skipped are exactly the lm_head
projection of RMSNorm(embedding row).  It is also checked against plain
arithmetic: an fp64 x @ W^T in numpy on the same bf16 weight bits, over
shapes that reach every path of the kernel (8-row and 16-row variants, no
split-K, split-K with a 16-wide remainder chunk, N not a multiple of 64).
Two calls in a row check that the shared scratch is reset between calls.
This file is collected last.
"""
import ctypes

import numpy as np
import pytest

import synth
from gpu_util import assert_logits_close

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def test_noalloc_projection_matches_decoder_logits():
    import paper_2309_08168_gb300 as ssd
    # d 1024 -> two 512-wide K chunks, so the split-K scratch is used;
    # vocab 4096 -> 64 row tiles
    w = synth.Workload("noalloc", 1, 1024, 8, 8, 128, 256, 4096, 4, 4, 1, 0, skip=[])
    hw = synth.host_weights(w, seed=3)
    dw = synth.host_to_device_weights(hw)
    torch.cuda.synchronize()
    cfg = ssd.make_config(w.n_layers, w.d_model, w.n_heads, w.n_kv_heads, w.head_dim, w.ffn, w.vocab, 32)
    dec = ssd.Decoder(cfg, dw, on_device=True)
    dec.set_skip(np.ones(2 * w.n_layers, np.uint8))
    M = 9
    toks = synth.prompt(M, seed=4, vocab=w.vocab)
    ref = dec.debug_forward(True, toks, 0)  # logits = W_head . RMSNorm(E[tok])

    e = synth.bf16_bits_to_f64(hw["embed"][toks]).astype(np.float32)
    x = e / np.sqrt((e * e).mean(axis=1, keepdims=True) + np.float32(w.rms_eps))
    x_dev = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    outs = []
    for _ in range(2):
        y = torch.full((M, w.vocab), float("nan"), dtype=torch.float32, device="cuda")
        torch.cuda.synchronize()
        rc = ssd.lib.ssd_linear_noalloc(dw["lm_head"].data_ptr(), x_dev.data_ptr(), y.data_ptr(),
                                        w.vocab, w.d_model, M, stream.cuda_stream)
        assert rc == ssd.SSD_OK, ssd.ssd_last_error()
        stream.synchronize()
        got = y.cpu().numpy()
        assert np.isfinite(got).all()
        assert_logits_close(got, ref, "no-alloc projection")
        outs.append(got)
    assert np.array_equal(outs[0].view(np.uint32), outs[1].view(np.uint32))
    dec.close()


@pytest.mark.parametrize("M,K,N", [(1, 528, 100), (8, 80, 64), (16, 4096, 4096), (9, 1024, 130)])
def test_noalloc_projection_matches_fp64_matmul(M, K, N):
    import paper_2309_08168_gb300 as ssd
    w_bits = synth.fill_bf16_host(N * K, seed=11, tid=900 + M, scale=1.0).reshape(N, K)
    rng = np.random.default_rng(M * 1000 + K)
    x = rng.standard_normal((M, K)).astype(np.float32)
    ref = x.astype(np.float64) @ synth.bf16_bits_to_f64(w_bits).T
    w_dev = torch.from_numpy(np.ascontiguousarray(w_bits).view(np.int16)).view(torch.bfloat16).cuda()
    x_dev = torch.from_numpy(x).cuda()
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    outs = []
    for _ in range(2):
        y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        torch.cuda.synchronize()
        rc = ssd.lib.ssd_linear_noalloc(w_dev.data_ptr(), x_dev.data_ptr(), y.data_ptr(), N, K, M,
                                        stream.cuda_stream)
        assert rc == ssd.SSD_OK, ssd.ssd_last_error()
        stream.synchronize()
        got = y.cpu().numpy()
        assert np.isfinite(got).all()
        assert_logits_close(got, ref, f"no-alloc projection M={M} K={K} N={N}")
        outs.append(got)
    assert np.array_equal(outs[0].view(np.uint32), outs[1].view(np.uint32))


def test_noalloc_rejects_oversized_problem():
    import paper_2309_08168_gb300 as ssd
    t = torch.zeros(16, dtype=torch.float32, device="cuda")
    rc = ssd.lib.ssd_linear_noalloc(t.data_ptr(), t.data_ptr(), t.data_ptr(), 32000, 8192, 16, None)
    assert rc == ssd.SSD_ERR_CAPACITY
    assert "scratch" in ssd.ssd_last_error()
