"""Seeded synthetic workloads for the self-speculative decoding path.

This module owns every input that the CUDA decode library and the fp64
oracle share: model shapes, skip masks, random-init bf16 weights and prompt
tokens.  It holds none of the decoding method's arithmetic.

Weights follow the recipe of the paper's LLaMA-2 evaluation models (Sec. 4.1,
App. B: LLaMA-2 7B/13B/70B in bf16) with random initialisation: every matrix
is N(0, 0.02) (Irwin-Hall(8) approximation, see synth_host.c), norm gains are
1.0, and the output projections of the sublayers the draft skips (Wo of a
skipped attention sublayer, Wd of a skipped MLP sublayer) are scaled by 0.05
before the single bf16 rounding, so that skipping them perturbs the residual
stream only a little and drafts are often accepted.

The host generator (C) and the device generator (CUDA) implement the same
definition; tests check they agree bit for bit.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_HOST_SO = os.path.join(_BUILD, "libsynth_host.so")
_DEV_SO = os.path.join(_BUILD, "libsynth_dev.so")

SIGMA = 0.02
SKIP_SCALE = 0.05
IH8_STD = 53509.91992145008  # std of a sum of 8 iid uniforms on {0..65535}

TID_EMBED = 0
TID_LM_HEAD = 1
_LAYER_NAMES = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")


def tensor_id(layer: int, name: str) -> int:
    return 16 + 8 * layer + _LAYER_NAMES.index(name)


def _stale(target, sources):
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(s) > t for s in sources)


def build_host() -> str:
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "synth_host.c")
    if _stale(_HOST_SO, [src]):
        tmp = _HOST_SO + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                               "-ffp-contract=off", src, "-o", tmp])
        os.replace(tmp, _HOST_SO)
    return _HOST_SO


def build_dev() -> str:
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "synth_dev.cu")
    if _stale(_DEV_SO, [src]):
        tmp = _DEV_SO + f".{os.getpid()}.tmp"
        subprocess.check_call(["nvcc", "-O3", "-std=c++17", "-shared", "-Xcompiler", "-fPIC",
                               "-gencode", "arch=compute_103a,code=sm_103a",
                               "-fmad=false", src, "-o", tmp])
        os.replace(tmp, _DEV_SO)
    return _DEV_SO


_host = None
_dev = None


def _host_lib():
    global _host
    if _host is None:
        lib = ctypes.CDLL(build_host())
        u64, u32, dbl = ctypes.c_uint64, ctypes.c_uint32, ctypes.c_double
        lib.synth_fill_bf16.argtypes = [ctypes.c_void_p, u64, u64, u64, u32, dbl]
        lib.synth_fill_f64.argtypes = [ctypes.c_void_p, u64, u64, u64, u32, dbl]
        lib.synth_prompt.argtypes = [ctypes.c_void_p, ctypes.c_int, u64, ctypes.c_int]
        lib.synth_round_bf16.argtypes = [ctypes.c_void_p, ctypes.c_void_p, u64]
        _host = lib
    return _host


def _dev_lib():
    global _dev
    if _dev is None:
        lib = ctypes.CDLL(build_dev())
        u64, u32, dbl = ctypes.c_uint64, ctypes.c_uint32, ctypes.c_double
        lib.synth_fill_bf16_dev.argtypes = [ctypes.c_void_p, u64, u64, u64, u32, dbl, ctypes.c_void_p]
        lib.synth_fill_bf16_dev.restype = ctypes.c_int
        lib.synth_fill_const_bf16_dev.argtypes = [ctypes.c_void_p, u64, ctypes.c_uint16, ctypes.c_void_p]
        lib.synth_fill_const_bf16_dev.restype = ctypes.c_int
        _dev = lib
    return _dev


def scale_const(scale: float) -> float:
    return SIGMA * scale / IH8_STD


def fill_bf16_host(n: int, seed: int, tid: int, scale: float = 1.0, first: int = 0) -> np.ndarray:
    out = np.empty(n, dtype=np.uint16)
    _host_lib().synth_fill_bf16(out.ctypes.data, first, n, seed, tid, scale_const(scale))
    return out


def fill_f64_host(n: int, seed: int, tid: int, scale: float = 1.0, first: int = 0) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    _host_lib().synth_fill_f64(out.ctypes.data, first, n, seed, tid, scale_const(scale))
    return out


def round_bf16_host(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(x.shape, dtype=np.uint16)
    _host_lib().synth_round_bf16(x.ctypes.data, out.ctypes.data, x.size)
    return out


def prompt(n: int, seed: int, vocab: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    _host_lib().synth_prompt(out.ctypes.data, n, seed, vocab)
    return out


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# Model shapes and workloads (LLaMA-2 shapes, Sec. 4.1; decoding settings of
# Table "Hyperparameter settings": T, K, top_p, temperature)
# ----------------------------------------------------------------------------

@dataclass
class Workload:
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    n_prompt: int
    n_new: int
    K: int
    mode: int  # 0 greedy, 1 sampling
    temperature: float = 1.0
    top_p: float = 1.0
    rms_eps: float = 1e-5
    rope_theta: float = 1e4
    skip: list = field(default_factory=list)  # skipped sublayer indices s = 2l + t

    @property
    def n_sublayers(self) -> int:
        return 2 * self.n_layers

    def mask(self) -> np.ndarray:
        m = np.zeros(self.n_sublayers, dtype=np.uint8)
        for s in self.skip:
            m[s] = 1
        return m

    def max_seq(self) -> int:
        return self.n_prompt + self.n_new + self.K + 1

    def truncated(self, n_layers: int, **kw) -> "Workload":
        """Same widths, fewer layers (skip window re-derived for the new depth)."""
        w = Workload(**{**self.__dict__, "n_layers": n_layers, "name": f"{self.name}-L{n_layers}"})
        w.skip = middle_window_skip(n_layers)
        for k, v in kw.items():
            setattr(w, k, v)
        return w


def middle_window_skip(n_layers: int) -> list:
    """Skip set for the LLaMA-shaped workloads: the contiguous window of
    sublayer indices s = 2l + t in [L/2, 3L/2) (t = 0 attention, 1 MLP), i.e.
    half of all sublayers, taken from the middle of the network and
    alternating attention / MLP inside the window."""
    return list(range(n_layers // 2, (3 * n_layers) // 2))


def workloads() -> dict:
    tiny = Workload("tiny", 4, 256, 4, 4, 64, 688, 2048, 32, 64, 4, 0, skip=[2, 5])
    w7 = Workload("llama2-7b", 32, 4096, 32, 32, 128, 11008, 32000, 512, 512, 8, 0,
                  skip=middle_window_skip(32))
    w13 = Workload("llama2-13b", 40, 5120, 40, 40, 128, 13824, 32000, 1024, 512, 8, 0,
                   skip=middle_window_skip(40))
    w13s = Workload("llama2-13b-sample", 40, 5120, 40, 40, 128, 13824, 32000, 1536, 512, 12, 1,
                    temperature=1.0, top_p=0.95, skip=middle_window_skip(40))
    w70 = Workload("llama2-70b", 80, 8192, 64, 8, 128, 28672, 32000, 1024, 256, 8, 0,
                   skip=middle_window_skip(80))
    return {w.name: w for w in (tiny, w7, w13, w13s, w70)}


def layer_scales(w: Workload, mask: np.ndarray) -> list:
    """Per layer (scale of Wo, scale of Wd)."""
    return [(SKIP_SCALE if mask[2 * l] else 1.0, SKIP_SCALE if mask[2 * l + 1] else 1.0)
            for l in range(w.n_layers)]


def tensor_shapes(w: Workload) -> dict:
    hq, hkv = w.n_heads * w.head_dim, w.n_kv_heads * w.head_dim
    return {"wq": (hq, w.d_model), "wk": (hkv, w.d_model), "wv": (hkv, w.d_model),
            "wo": (w.d_model, hq), "w_gate": (w.ffn, w.d_model), "w_up": (w.ffn, w.d_model),
            "w_down": (w.d_model, w.ffn)}


ONE_BF16 = 0x3F80


def host_weights(w: Workload, seed: int, mask: np.ndarray | None = None) -> dict:
    """All weights as host bf16 bit arrays (numpy uint16), row-major [out][in]."""
    if mask is None:
        mask = w.mask()
    shapes = tensor_shapes(w)
    sc = layer_scales(w, mask)
    out = {
        "embed": fill_bf16_host(w.vocab * w.d_model, seed, TID_EMBED).reshape(w.vocab, w.d_model),
        "lm_head": fill_bf16_host(w.vocab * w.d_model, seed, TID_LM_HEAD).reshape(w.vocab, w.d_model),
        "final_norm": np.full(w.d_model, ONE_BF16, dtype=np.uint16),
        "layers": [],
    }
    for l in range(w.n_layers):
        layer = {"attn_norm": np.full(w.d_model, ONE_BF16, dtype=np.uint16),
                 "mlp_norm": np.full(w.d_model, ONE_BF16, dtype=np.uint16)}
        for name, shp in shapes.items():
            s = sc[l][0] if name == "wo" else (sc[l][1] if name == "w_down" else 1.0)
            layer[name] = fill_bf16_host(shp[0] * shp[1], seed, tensor_id(l, name), s).reshape(shp)
        out["layers"].append(layer)
    return out


def device_weights(w: Workload, seed: int, mask: np.ndarray | None = None, device="cuda"):
    """All weights as bf16 torch tensors in HBM, written by the device generator."""
    import torch
    if mask is None:
        mask = w.mask()
    lib = _dev_lib()
    stream = torch.cuda.current_stream(device).cuda_stream
    shapes = tensor_shapes(w)
    sc = layer_scales(w, mask)

    def gen(shape, tid, scale=1.0):
        t = torch.empty(shape, dtype=torch.bfloat16, device=device)
        rc = lib.synth_fill_bf16_dev(t.data_ptr(), 0, t.numel(), seed, tid, scale_const(scale), stream)
        if rc != 0:
            raise RuntimeError(f"synth device fill failed: cuda error {rc}")
        return t

    def ones(n):
        t = torch.empty(n, dtype=torch.bfloat16, device=device)
        rc = lib.synth_fill_const_bf16_dev(t.data_ptr(), n, ONE_BF16, stream)
        if rc != 0:
            raise RuntimeError(f"synth device fill failed: cuda error {rc}")
        return t

    out = {"embed": gen((w.vocab, w.d_model), TID_EMBED),
           "lm_head": gen((w.vocab, w.d_model), TID_LM_HEAD),
           "final_norm": ones(w.d_model), "layers": []}
    for l in range(w.n_layers):
        layer = {"attn_norm": ones(w.d_model), "mlp_norm": ones(w.d_model)}
        for name, shp in shapes.items():
            s = sc[l][0] if name == "wo" else (sc[l][1] if name == "w_down" else 1.0)
            layer[name] = gen(shp, tensor_id(l, name), s)
        out["layers"].append(layer)
    return out


def host_to_device_weights(hw: dict, device="cuda"):
    """Upload host bf16 bit arrays as torch bf16 tensors (same bits)."""
    import torch

    def up(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)

    return {"embed": up(hw["embed"]), "lm_head": up(hw["lm_head"]), "final_norm": up(hw["final_norm"]),
            "layers": [{k: up(v) for k, v in layer.items()} for layer in hw["layers"]]}


def weight_bytes(w: Workload, mask: np.ndarray | None = None, draft: bool = False) -> int:
    """Algorithmic weight bytes one forward streams from HBM (bf16): every
    matrix of every sublayer that runs, the norm gains, one embedding row and
    the whole lm_head.  With draft=True the sublayers in `mask` are skipped."""
    if mask is None:
        mask = w.mask()
    hq, hkv = w.n_heads * w.head_dim, w.n_kv_heads * w.head_dim
    attn = (hq * w.d_model + 2 * hkv * w.d_model + w.d_model * hq + w.d_model) * 2
    mlp = (3 * w.ffn * w.d_model + w.d_model) * 2
    total = (w.d_model + w.vocab * w.d_model + w.d_model) * 2
    for l in range(w.n_layers):
        if not (draft and mask[2 * l]):
            total += attn
        if not (draft and mask[2 * l + 1]):
            total += mlp
    return total


def kv_bytes_read(w: Workload, ctx: int, mask: np.ndarray | None = None, draft: bool = False) -> int:
    """KV-cache bytes one forward reads at context length ctx (bf16 K and V)."""
    if mask is None:
        mask = w.mask()
    per_layer = 2 * w.n_kv_heads * w.head_dim * 2 * ctx
    n_attn = sum(1 for l in range(w.n_layers) if not (draft and mask[2 * l]))
    return per_layer * n_attn
