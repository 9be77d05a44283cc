"""Python binding of libssd, batch-1 self-speculative decoding on GB300.

Argument marshalling only: every step of the decode path runs in the CUDA
library (csrc/, built for sm_103a by build.py).  The functions keep the C
ABI's names (include/ssd.h).  Importing this module fails loudly when the
library has not been built; there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libssd.so")

SSD_OK = 0
SSD_ERR_INVALID_ARG = -1
SSD_ERR_OOM = -2
SSD_ERR_CUDA = -3
SSD_ERR_CAPACITY = -4
SSD_ERR_TIMEOUT = -5
SSD_ERR_STATE = -6
SSD_GREEDY = 0
SSD_SAMPLE = 1

# every symbol include/ssd.h declares
EXPORTS = ("ssd_create", "ssd_set_skip", "ssd_set_sampling", "ssd_set_draft_exit", "ssd_prefill", "ssd_generate",
           "ssd_debug_forward", "ssd_debug_spec_accept", "ssd_debug_time_forward", "ssd_destroy",
           "ssd_last_error", "ssd_linear_noalloc", "ssd_debug_trace_forward", "ssd_debug_stall_barrier")


class ssd_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in
                ("n_layers", "d_model", "n_heads", "n_kv_heads", "head_dim", "ffn", "vocab", "max_seq")] + \
               [("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)]


_VP = ctypes.c_void_p
_VPP = ctypes.POINTER(ctypes.c_void_p)
LAYER_TENSORS = ("wq", "wk", "wv", "wo", "attn_norm", "w_gate", "w_up", "w_down", "mlp_norm")


class ssd_weights(ctypes.Structure):
    _fields_ = [("embed", _VP), ("final_norm", _VP), ("lm_head", _VP)] + \
               [(n, _VPP) for n in LAYER_TENSORS] + [("on_device", ctypes.c_int)]


class ssd_stats(ctypes.Structure):
    _fields_ = [("rounds", ctypes.c_int), ("drafted", ctypes.c_int), ("accepted", ctypes.c_int),
                ("emitted", ctypes.c_int), ("accept_rate", ctypes.c_double), ("hist", ctypes.c_int * 33),
                ("draft_ms", ctypes.c_float), ("verify_ms", ctypes.c_float), ("total_ms", ctypes.c_float),
                ("kernel_launches", ctypes.c_longlong), ("gamma", ctypes.c_float)]

    def as_dict(self) -> dict:
        return {"rounds": self.rounds, "drafted": self.drafted, "accepted": self.accepted,
                "emitted": self.emitted, "accept_rate": self.accept_rate, "hist": list(self.hist),
                "draft_ms": self.draft_ms, "verify_ms": self.verify_ms, "total_ms": self.total_ms,
                "kernel_launches": self.kernel_launches, "gamma": self.gamma}


class SSDError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{msg} (code {code})")
        self.code = code


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libssd is not built ({LIB_PATH} missing); run "
                          "`python -c 'import __graft_entry__ as g; g.build()'` first")
    lib = ctypes.CDLL(LIB_PATH)
    H = ctypes.c_void_p
    lib.ssd_create.argtypes = [ctypes.POINTER(ssd_config), ctypes.POINTER(ssd_weights), _VP, ctypes.POINTER(H)]
    lib.ssd_set_skip.argtypes = [H, _VP, ctypes.c_int]
    lib.ssd_set_sampling.argtypes = [H, ctypes.c_float, ctypes.c_float]
    lib.ssd_set_draft_exit.argtypes = [H, ctypes.c_int] + [ctypes.c_float] * 5
    lib.ssd_prefill.argtypes = [H, _VP, ctypes.c_int]
    lib.ssd_generate.argtypes = [H, _VP, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                 ctypes.c_uint64, _VP, ctypes.POINTER(ssd_stats)]
    lib.ssd_debug_forward.argtypes = [H, ctypes.c_int, _VP, ctypes.c_int, ctypes.c_int, _VP]
    lib.ssd_debug_spec_accept.argtypes = [H, _VP, _VP, ctypes.c_int, _VP, _VP, ctypes.c_int, ctypes.c_int, _VP]
    lib.ssd_debug_time_forward.argtypes = [H, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                           _VP, _VP, _VP]
    lib.ssd_debug_trace_forward.argtypes = [H, ctypes.c_int, ctypes.c_int, _VP, _VP, ctypes.c_int, _VP,
                                            ctypes.c_int, _VP, _VP, ctypes.c_int, _VP]
    lib.ssd_debug_trace_forward.restype = ctypes.c_int
    lib.ssd_debug_stall_barrier.argtypes = [H, ctypes.c_int, ctypes.c_double]
    lib.ssd_debug_stall_barrier.restype = ctypes.c_int
    lib.ssd_linear_noalloc.argtypes = [_VP, _VP, _VP, ctypes.c_int, ctypes.c_int, ctypes.c_int, _VP]
    lib.ssd_linear_noalloc.restype = ctypes.c_int
    lib.ssd_destroy.argtypes = [H]
    lib.ssd_destroy.restype = None
    lib.ssd_last_error.argtypes = []
    lib.ssd_last_error.restype = ctypes.c_char_p
    for n in ("ssd_create", "ssd_set_skip", "ssd_set_sampling", "ssd_set_draft_exit", "ssd_prefill",
              "ssd_generate", "ssd_debug_forward", "ssd_debug_spec_accept", "ssd_debug_time_forward"):
        getattr(lib, n).restype = ctypes.c_int
    return lib


lib = _load()


def _check(rc: int):
    if rc != SSD_OK:
        raise SSDError(rc, lib.ssd_last_error().decode())


def _ptr(a) -> int:
    """Address of a numpy array or a torch tensor."""
    if hasattr(a, "data_ptr"):
        return a.data_ptr()
    return a.ctypes.data


# -- the C ABI, one function each -------------------------------------------

def ssd_create(cfg: ssd_config, weights: ssd_weights, cuda_stream: int | None = None) -> int:
    h = ctypes.c_void_p()
    _check(lib.ssd_create(ctypes.byref(cfg), ctypes.byref(weights), cuda_stream, ctypes.byref(h)))
    _configs[h.value] = cfg
    return h.value


def ssd_set_skip(h: int, mask) -> None:
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    _check(lib.ssd_set_skip(h, m.ctypes.data, m.size))


def ssd_set_sampling(h: int, temperature: float, top_p: float) -> None:
    _check(lib.ssd_set_sampling(h, temperature, top_p))


def ssd_set_draft_exit(h: int, enable: bool, gamma0: float = 0.6, alpha: float = 0.9, eps: float = 0.01,
                       beta1: float = 0.5, beta2: float = 0.9) -> None:
    _check(lib.ssd_set_draft_exit(h, int(bool(enable)), gamma0, alpha, eps, beta1, beta2))


def ssd_prefill(h: int, prompt) -> None:
    p = np.ascontiguousarray(prompt, dtype=np.int32)
    _check(lib.ssd_prefill(h, p.ctypes.data, p.size))


def ssd_generate(h: int, prompt, n_new: int, K: int, mode: int = SSD_GREEDY, seed: int = 0,
                 out=None):
    """prompt: host int32 tokens or None (restart from the last prefill).
    Returns (tokens np.int32[n_new], stats dict)."""
    if prompt is None:
        pp, pn = None, 0
    else:
        p = np.ascontiguousarray(prompt, dtype=np.int32)
        pp, pn = p.ctypes.data, p.size
    toks = out if out is not None else np.zeros(n_new, dtype=np.int32)
    st = ssd_stats()
    _check(lib.ssd_generate(h, pp, pn, n_new, K, mode, seed, _ptr(toks) if n_new else None, ctypes.byref(st)))
    return toks, st.as_dict()


def ssd_debug_forward(h: int, draft: bool, tokens, pos0: int) -> np.ndarray:
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    out = np.empty((t.size, config_of(h).vocab), dtype=np.float32)
    _check(lib.ssd_debug_forward(h, int(draft), t.ctypes.data, t.size, pos0, out.ctypes.data))
    return out


def ssd_debug_stall_barrier(h: int, barrier: int, wait_limit_s: float) -> None:
    _check(lib.ssd_debug_stall_barrier(h, int(barrier), float(wait_limit_s)))


def ssd_debug_spec_accept(h: int, p, q, drafts, seeds, pos0: int):
    p = np.ascontiguousarray(p, dtype=np.float32)
    q = np.ascontiguousarray(q, dtype=np.float32)
    d = np.ascontiguousarray(drafts, dtype=np.int32)
    s = np.ascontiguousarray(seeds, dtype=np.uint64)
    T, Kd = d.shape
    out = np.empty((T, 2), dtype=np.int32)
    _check(lib.ssd_debug_spec_accept(h, p.ctypes.data, q.ctypes.data, Kd, d.ctypes.data, s.ctypes.data,
                                     T, pos0, out.ctypes.data))
    return out[:, 0], out[:, 1]


def ssd_debug_time_forward(h: int, draft: bool, rows: int, gemm_only: bool, reps: int):
    """Returns (ms per forward replay, kernels per replay, weight bytes per replay)."""
    ms = ctypes.c_float()
    n = ctypes.c_int()
    b = ctypes.c_double()
    _check(lib.ssd_debug_time_forward(h, int(draft), rows, int(gemm_only), reps, ctypes.addressof(ms),
                                      ctypes.addressof(n), ctypes.addressof(b)))
    return ms.value, n.value, b.value


def ssd_linear_noalloc(w, x, y, N: int, K: int, M: int, cuda_stream: int | None = None) -> None:
    """y[M][N] = x[M][K] @ w[N][K]^T on device tensors, without allocating."""
    _check(lib.ssd_linear_noalloc(_ptr(w), _ptr(x), _ptr(y), N, K, M, cuda_stream))


OP_NAMES = ("embed", "qkv", "attention", "o/down", "gate/up", "lm_head")


def ssd_debug_trace_forward(h: int, draft: bool, rows: int, detail_op: int = -1):
    """Returns [(op name, microseconds)] for one forward of the forward kernel.
    With detail_op >= 0 (op index + 65536 x a CTA index) it returns (ops,
    units, ctas): units = [64][4] stamps (ns) of that CTA's first work units
    of that op (producer issue, MMAs issued, 0, segment flush done; for
    attention 8 stamps per item), ctas = [grid][8] stamps per CTA in the
    order ssd.h lists."""
    cfg = config_of(h)
    cap = 2 + 5 * cfg.n_layers
    us = np.zeros(cap, dtype=np.float32)
    ty = np.zeros(cap, dtype=np.int32)
    ut = np.zeros((64, 4), dtype=np.uint64)
    max_ctas = 1024
    ct = np.zeros((max_ctas, 8), dtype=np.uint64)
    n = ctypes.c_int()
    n_ctas = ctypes.c_int()
    detail = detail_op >= 0
    _check(lib.ssd_debug_trace_forward(h, int(draft), rows, us.ctypes.data, ty.ctypes.data, cap,
                                       ctypes.addressof(n), int(detail_op), ut.ctypes.data if detail else None,
                                       ct.ctypes.data if detail else None, max_ctas, ctypes.addressof(n_ctas)))
    ops = [(OP_NAMES[ty[i]], float(us[i])) for i in range(n.value)]
    return (ops, ut, ct[:n_ctas.value]) if detail else ops


def ssd_destroy(h: int) -> None:
    if h:
        _configs.pop(h, None)
        lib.ssd_destroy(h)


def ssd_last_error() -> str:
    return lib.ssd_last_error().decode()


# -- marshalling helpers -----------------------------------------------------

_configs: dict = {}


def config_of(h: int) -> ssd_config:
    return _configs[h]


def make_config(n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab, max_seq,
                rms_eps=1e-5, rope_theta=1e4) -> ssd_config:
    return ssd_config(n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab, max_seq,
                      rms_eps, rope_theta)


class WeightRefs:
    """ssd_weights built from a dict {embed, final_norm, lm_head, layers:[{wq..}]}
    of torch tensors (on_device=1) or numpy arrays (on_device=0).  Keeps the
    pointer arrays alive."""

    def __init__(self, weights: dict, on_device: bool):
        L = len(weights["layers"])
        self.keep = [weights]
        self.struct = ssd_weights()
        self.struct.embed = _ptr(weights["embed"])
        self.struct.final_norm = _ptr(weights["final_norm"])
        self.struct.lm_head = _ptr(weights["lm_head"])
        for name in LAYER_TENSORS:
            arr = (ctypes.c_void_p * L)(*[_ptr(layer[name]) for layer in weights["layers"]])
            self.keep.append(arr)
            setattr(self.struct, name, ctypes.cast(arr, _VPP))
        self.struct.on_device = 1 if on_device else 0


class Decoder:
    """Owns one ssd handle (thin convenience wrapper over the C ABI)."""

    def __init__(self, cfg: ssd_config, weights: dict, on_device: bool = True, stream: int | None = None):
        self.cfg = cfg
        self.refs = WeightRefs(weights, on_device)
        self.h = ssd_create(cfg, self.refs.struct, stream)

    def close(self):
        if self.h:
            ssd_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_skip(self, mask):
        ssd_set_skip(self.h, mask)

    def set_sampling(self, temperature, top_p):
        ssd_set_sampling(self.h, temperature, top_p)

    def set_draft_exit(self, enable, gamma0=0.6, alpha=0.9, eps=0.01, beta1=0.5, beta2=0.9):
        ssd_set_draft_exit(self.h, enable, gamma0, alpha, eps, beta1, beta2)

    def prefill(self, prompt):
        ssd_prefill(self.h, prompt)

    def generate(self, prompt, n_new, K, mode=SSD_GREEDY, seed=0, out=None):
        return ssd_generate(self.h, prompt, n_new, K, mode, seed, out)

    def debug_forward(self, draft, tokens, pos0):
        return ssd_debug_forward(self.h, draft, tokens, pos0)

    def debug_stall_barrier(self, barrier, wait_limit_s):
        return ssd_debug_stall_barrier(self.h, barrier, wait_limit_s)

    def debug_spec_accept(self, p, q, drafts, seeds, pos0):
        return ssd_debug_spec_accept(self.h, p, q, drafts, seeds, pos0)

    def debug_time_forward(self, draft, rows, gemm_only, reps):
        return ssd_debug_time_forward(self.h, draft, rows, gemm_only, reps)

    def debug_trace_forward(self, draft, rows, detail_op=-1):
        return ssd_debug_trace_forward(self.h, draft, rows, detail_op)
