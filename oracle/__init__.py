"""fp64 CPU oracle for self-speculative decoding (arxiv 2309.08168).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline leg of bench.py, never by the decode library.  It shares no code
with the CUDA path.  The arithmetic lives in oracle.c (plain C, fp64); this
file compiles it and marshals arguments.

Parity status per function (pins are in tests/test_oracle_*.py):
  orc_forward / orc_forward_uncached  pinned: torch-fp64 library composition,
                                      cache == brute force, closed forms
  orc_generate greedy (Alg. 1 / 2)    pinned: lossless invariant SSD == AR,
                                      empty mask => every draft accepted
  orc_generate sampling (Alg. 4)      pinned through orc_spec_verify's exact
                                      output law and the empty-mask case
  orc_spec_verify                     pinned: output law integrates to p
  orc_nucleus_probs / orc_sample      pinned: hand-worked golden cases
  orc_philox4x32_10                   pinned: published known-answer vectors
  orc_exit_update (Eqs. 2-4)          pinned: closed forms of the gamma / AR
                                      recurrences (constant and alternating AR_e)
  orc_generate_ex (draft exit,        pinned: gamma = 0 reproduces no exit,
    Algs. 3 / 4)                      gamma > 1 drafts once per round, lossless
                                      invariant SSD == AR with exit
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")


def build() -> str:
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "oracle.c")
    if not os.path.exists(_SO) or os.path.getmtime(src) > os.path.getmtime(_SO):
        tmp = _SO + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                               "-ffp-contract=off", src, "-o", tmp, "-lm"])
        os.replace(tmp, _SO)
    return _SO


class OrcConfig(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in
                ("n_layers", "d_model", "n_heads", "n_kv_heads", "head_dim", "ffn", "vocab", "max_seq")] + \
               [("rms_eps", ctypes.c_double), ("rope_theta", ctypes.c_double)]


_P = ctypes.c_void_p
_PP = ctypes.POINTER(ctypes.c_void_p)


class OrcWeights(ctypes.Structure):
    _fields_ = [("embed", _P), ("final_norm", _P), ("lm_head", _P)] + \
               [(n, _PP) for n in ("wq", "wk", "wv", "wo", "attn_norm", "w_gate", "w_up", "w_down", "mlp_norm")]


class OrcExit(ctypes.Structure):
    _fields_ = [("on", ctypes.c_int)] + [(n, ctypes.c_double) for n in ("gamma0", "alpha", "eps", "beta1", "beta2")]


class OrcExitState(ctypes.Structure):
    _fields_ = [("gamma", ctypes.c_double), ("ar", ctypes.c_double), ("e", ctypes.c_int)]


class OrcStats(ctypes.Structure):
    _fields_ = [("rounds", ctypes.c_int), ("drafted", ctypes.c_int), ("accepted", ctypes.c_int),
                ("emitted", ctypes.c_int), ("hist", ctypes.c_int * 33)]


_lib = None


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        L.orc_create.argtypes = [ctypes.POINTER(OrcConfig), ctypes.POINTER(OrcWeights)]
        L.orc_create.restype = _P
        L.orc_destroy.argtypes = [_P]
        L.orc_cache.argtypes = [_P, ctypes.c_int]
        L.orc_cache.restype = ctypes.POINTER(ctypes.c_double)
        L.orc_forward.argtypes = [_P, ctypes.c_int, ctypes.c_int, _P, _P]
        L.orc_forward_uncached.argtypes = [_P, _P, ctypes.c_int, ctypes.c_int, _P, _P]
        L.orc_forward_uncached.restype = ctypes.c_int
        L.orc_prefill.argtypes = [_P, _P, ctypes.c_int]
        L.orc_prefill.restype = ctypes.c_int
        L.orc_generate.argtypes = [_P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                   ctypes.c_uint64, ctypes.c_double, ctypes.c_double, _P, _P,
                                   ctypes.POINTER(OrcStats), _P, _P]
        L.orc_generate.restype = ctypes.c_int
        L.orc_generate_ex.argtypes = L.orc_generate.argtypes + [ctypes.POINTER(OrcExit), _P, _P]
        L.orc_generate_ex.restype = ctypes.c_int
        L.orc_exit_update.argtypes = [ctypes.POINTER(OrcExitState), ctypes.POINTER(OrcExit), ctypes.c_double]
        L.orc_softmax_max.argtypes = [_P, ctypes.c_int]
        L.orc_softmax_max.restype = ctypes.c_double
        L.orc_set_threads.argtypes = [ctypes.c_int]
        L.orc_get_threads.restype = ctypes.c_int
        L.orc_rmsnorm.argtypes = [_P, _P, ctypes.c_int, ctypes.c_double, _P]
        L.orc_rope.argtypes = [_P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double]
        L.orc_philox4x32_10.argtypes = [_P, _P, _P]
        L.orc_uniform.argtypes = [ctypes.c_uint64, ctypes.c_int, ctypes.c_int]
        L.orc_uniform.restype = ctypes.c_double
        L.orc_argmax.argtypes = [_P, ctypes.c_int]
        L.orc_argmax.restype = ctypes.c_int
        L.orc_nucleus_probs.argtypes = [_P, ctypes.c_int, ctypes.c_double, ctypes.c_double, _P]
        L.orc_sample.argtypes = [_P, ctypes.c_int, ctypes.c_double]
        L.orc_sample.restype = ctypes.c_int
        L.orc_spec_verify.argtypes = [_P, _P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P]
        L.orc_spec_verify.restype = ctypes.c_int
        L.orc_spec_verify_batch.argtypes = [_P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P]
        _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


class Oracle:
    """One fp64 model instance over host bf16 weights (numpy uint16 arrays).

    `weights` is the dict layout produced by synth.host_weights; the arrays
    must stay alive as long as this object (it keeps a reference)."""

    def __init__(self, w, weights: dict, max_seq: int):
        self.w = w
        self.weights = weights
        self.max_seq = max_seq
        L = len(weights["layers"])
        self.n_layers = L
        self.cfg = OrcConfig(L, w.d_model, w.n_heads, w.n_kv_heads, w.head_dim, w.ffn, w.vocab,
                             max_seq, w.rms_eps, w.rope_theta)
        self._arrays = {}
        ow = OrcWeights()
        ow.embed = _ptr(weights["embed"])
        ow.final_norm = _ptr(weights["final_norm"])
        ow.lm_head = _ptr(weights["lm_head"])
        for name in ("wq", "wk", "wv", "wo", "attn_norm", "w_gate", "w_up", "w_down", "mlp_norm"):
            arr = (ctypes.c_void_p * L)(*[_ptr(layer[name]) for layer in weights["layers"]])
            self._arrays[name] = arr
            setattr(ow, name, ctypes.cast(arr, _PP))
        self._ow = ow
        self.h = lib().orc_create(ctypes.byref(self.cfg), ctypes.byref(ow))
        if not self.h:
            raise ValueError("orc_create rejected the configuration")

    def close(self):
        if self.h:
            lib().orc_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _mask(self, mask):
        if mask is None:
            return None
        m = np.ascontiguousarray(mask, dtype=np.uint8)
        assert m.size == 2 * self.n_layers
        return m

    def forward(self, tok: int, pos: int, mask=None, want_logits=True):
        m = self._mask(mask)
        out = np.empty(self.w.vocab, dtype=np.float64) if want_logits else None
        lib().orc_forward(self.h, int(tok), int(pos), None if m is None else _ptr(m),
                          None if out is None else _ptr(out))
        return out

    def forward_uncached(self, toks, n_full=None, mask=None):
        t = np.ascontiguousarray(toks, dtype=np.int32)
        n = t.size
        n_full = n if n_full is None else n_full
        m = self._mask(mask)
        out = np.empty((n, self.w.vocab), dtype=np.float64)
        rc = lib().orc_forward_uncached(self.h, _ptr(t), n, n_full, None if m is None else _ptr(m), _ptr(out))
        if rc:
            raise ValueError("orc_forward_uncached: bad arguments")
        return out

    def prefill(self, prompt):
        p = np.ascontiguousarray(prompt, dtype=np.int32)
        if lib().orc_prefill(self.h, _ptr(p), p.size):
            raise ValueError("orc_prefill: bad arguments")

    def cache(self, which: int) -> np.ndarray:
        ptr = lib().orc_cache(self.h, which)
        n = self.n_layers * self.max_seq * self.w.n_kv_heads * self.w.head_dim
        return np.ctypeslib.as_array(ptr, shape=(n,)).reshape(
            self.n_layers, self.max_seq, self.w.n_kv_heads * self.w.head_dim)

    def generate(self, prompt, n_new: int, K: int, mode: int = 0, seed: int = 0,
                 temperature: float = 1.0, top_p: float = 1.0, mask=None, want_logits=False,
                 draft_exit=None):
        """draft_exit: None, or (gamma0, alpha, eps, beta1, beta2) of the
        adaptive draft exit; stats then also hold every round's draft count
        ("keff") and gamma after its update ("gamma")."""
        p = np.ascontiguousarray(prompt, dtype=np.int32)
        m = self._mask(mask)
        out = np.zeros(n_new, dtype=np.int32)
        st = OrcStats()
        dl = vl = None
        if want_logits:
            dl = np.zeros((max(K, 1), self.w.vocab), dtype=np.float64)
            vl = np.zeros((K + 1, self.w.vocab), dtype=np.float64)
        ex = OrcExit(0, 0.0, 0.0, 0.0, 0.0, 0.0) if draft_exit is None else OrcExit(1, *map(float, draft_exit))
        keff = np.zeros(max(n_new, 1), dtype=np.int32)
        gam = np.zeros(max(n_new, 1), dtype=np.float64)
        rc = lib().orc_generate_ex(self.h, _ptr(p), p.size, n_new, K, mode, seed, temperature, top_p,
                                   None if m is None else _ptr(m), _ptr(out), ctypes.byref(st),
                                   None if dl is None else _ptr(dl), None if vl is None else _ptr(vl),
                                   ctypes.byref(ex), _ptr(keff), _ptr(gam))
        if rc:
            raise ValueError(f"orc_generate failed ({rc})")
        stats = {"rounds": st.rounds, "drafted": st.drafted, "accepted": st.accepted,
                 "emitted": st.emitted, "hist": list(st.hist),
                 "keff": keff[:st.rounds].tolist(), "gamma": gam[:st.rounds].tolist()}
        if want_logits:
            return out, stats, dl, vl
        return out, stats


# -- stateless helpers ------------------------------------------------------

def rmsnorm(x, g_bits, eps):
    x = np.ascontiguousarray(x, dtype=np.float64)
    g = np.ascontiguousarray(g_bits, dtype=np.uint16)
    out = np.empty_like(x)
    lib().orc_rmsnorm(_ptr(x), _ptr(g), x.size, eps, _ptr(out))
    return out


def rope(v, n_heads, head_dim, pos, theta):
    v = np.array(v, dtype=np.float64, copy=True)
    lib().orc_rope(_ptr(v), n_heads, head_dim, pos, theta)
    return v


def philox(ctr, key):
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def uniform(seed, pos, purpose):
    return lib().orc_uniform(seed, pos, purpose)


def argmax(x):
    x = np.ascontiguousarray(x, dtype=np.float64)
    return lib().orc_argmax(_ptr(x), x.size)


def nucleus_probs(logits, temperature, top_p):
    x = np.ascontiguousarray(logits, dtype=np.float64)
    out = np.empty_like(x)
    lib().orc_nucleus_probs(_ptr(x), x.size, temperature, top_p, _ptr(out))
    return out


def sample(probs, u):
    p = np.ascontiguousarray(probs, dtype=np.float64)
    return lib().orc_sample(_ptr(p), p.size, u)


def spec_verify(p_rows, q_rows, drafts, r, ures):
    p = np.ascontiguousarray(p_rows, dtype=np.float64)
    q = np.ascontiguousarray(q_rows, dtype=np.float64)
    d = np.ascontiguousarray(drafts, dtype=np.int32)
    rr = np.ascontiguousarray(r, dtype=np.float64)
    uu = np.ascontiguousarray(ures, dtype=np.float64)
    n = ctypes.c_int(0)
    y = lib().orc_spec_verify(_ptr(p), _ptr(q), _ptr(d), d.size, p.shape[1], _ptr(rr), _ptr(uu),
                              ctypes.addressof(n))
    return n.value, y


def spec_verify_batch(p_rows, q_rows, drafts, r, ures):
    """drafts: [T][Kd]; r: [T][Kd]; ures: [T][Kd+1] -> (n[T], y[T])."""
    p = np.ascontiguousarray(p_rows, dtype=np.float64)
    q = np.ascontiguousarray(q_rows, dtype=np.float64)
    d = np.ascontiguousarray(drafts, dtype=np.int32)
    rr = np.ascontiguousarray(r, dtype=np.float64)
    uu = np.ascontiguousarray(ures, dtype=np.float64)
    T, Kd = d.shape
    out = np.empty((T, 2), dtype=np.int32)
    lib().orc_spec_verify_batch(_ptr(p), _ptr(q), Kd, p.shape[1], T, _ptr(d), _ptr(rr), _ptr(uu), _ptr(out))
    return out[:, 0], out[:, 1]


def exit_update(state, params, ar_e):
    """One application of Eqs. 2-4: state = (gamma, ar, e), params = (gamma0,
    alpha, eps, beta1, beta2); returns the new state."""
    st = OrcExitState(*state)
    lib().orc_exit_update(ctypes.byref(st), ctypes.byref(OrcExit(1, *map(float, params))), float(ar_e))
    return st.gamma, st.ar, st.e


def set_threads(n: int) -> None:
    """OpenMP threads of the oracle (timing only; results do not depend on it)."""
    lib().orc_set_threads(int(n))


def get_threads() -> int:
    return int(lib().orc_get_threads())


def softmax_max(logits):
    x = np.ascontiguousarray(logits, dtype=np.float64)
    return lib().orc_softmax_max(_ptr(x), x.size)
