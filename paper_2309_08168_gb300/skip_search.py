"""Search for the draft model's skip set z (Sec. 3.3).

The paper picks z* = argmin_z f(z), f = average inference time per verified
(emitted) token on a development set, with Bayesian optimisation.  This
module keeps the objective and replaces the optimiser by a local search that
needs no third-party library: starting from a mask, it proposes single-bit
flips of z (skip one more sublayer, or run one that was skipped), evaluates
each proposal on the GPU through the decoder and keeps it when f improves.

f is measured, so it carries timing noise; the search therefore re-measures
the incumbent whenever it would accept a proposal by less than `rel_margin`.

Host logic only: every forward, draft and acceptance runs in the library.
"""
from __future__ import annotations

from typing import Callable, Sequence

import numpy as np


def ms_per_token(dec, prompts: Sequence[np.ndarray], n_new: int, K: int, mode: int = 0,
                 seed: int = 0) -> float:
    """f(z) for the decoder's current skip set: GPU time of the decoding
    loops (prefill excluded) over the development prompts, divided by the
    tokens they emitted, in ms."""
    total_ms = 0.0
    tokens = 0
    for p in prompts:
        dec.prefill(p)
        _, st = dec.generate(None, n_new, K, mode=mode, seed=seed)
        total_ms += st["total_ms"]
        tokens += st["emitted"]
    return total_ms / max(tokens, 1)


class Objective:
    """Memoised f over masks (a mask is measured once unless re-measured)."""

    def __init__(self, measure: Callable[[np.ndarray], float]):
        self.measure = measure
        self.cache: dict[bytes, float] = {}
        self.evals = 0

    def __call__(self, mask: np.ndarray, fresh: bool = False) -> float:
        key = np.asarray(mask, dtype=np.uint8).tobytes()
        if fresh or key not in self.cache:
            self.evals += 1
            v = float(self.measure(np.asarray(mask, dtype=np.uint8)))
            # several measurements of one mask: keep the smallest (timing noise is one-sided)
            self.cache[key] = min(v, self.cache.get(key, v))
        return self.cache[key]


def local_search(f: Objective, start: np.ndarray, budget: int, rng: np.random.Generator,
                 allowed: Sequence[int] | None = None, rel_margin: float = 0.01,
                 max_skip: int | None = None):
    """Stochastic first-improvement hill climbing over single-bit flips of z.

    f: objective over uint8 masks; start: initial mask; budget: measurements
    allowed (re-measurements included); allowed: sublayer indices that may
    change (default all); max_skip: upper bound on the number of skipped
    sublayers.  Each pass visits the allowed indices in a random order.
    Returns (best mask, its f, history of (mask bits, f, accepted))."""
    z = np.array(start, dtype=np.uint8)
    idx = list(range(z.size)) if allowed is None else list(allowed)
    best = f(z)
    history = [(z.copy(), best, True)]
    improved = True
    while improved and f.evals < budget:
        improved = False
        for i in rng.permutation(idx):
            if f.evals >= budget:
                break
            cand = z.copy()
            cand[i] ^= 1
            if max_skip is not None and int(cand.sum()) > max_skip:
                continue
            v = f(cand)
            accept = v < best
            if accept and v > best * (1.0 - rel_margin) and f.evals < budget:
                best = min(best, f(z, fresh=True))  # a narrow win: confirm against a fresh incumbent
                accept = v < best
            history.append((cand.copy(), v, bool(accept)))
            if accept:
                z, best, improved = cand, v, True
    return z, best, history


def search_skip_set(dec, prompts, n_new: int, K: int, start: np.ndarray, budget: int = 40, seed: int = 0,
                    mode: int = 0, allowed=None, max_skip=None):
    """Runs local_search with f = ms_per_token on the decoder; leaves the
    decoder's skip set at the best mask found.  Returns (mask, f, history,
    f(start))."""
    def measure(mask):
        dec.set_skip(mask)
        return ms_per_token(dec, prompts, n_new, K, mode=mode, seed=seed)

    f = Objective(measure)
    f0 = f(np.asarray(start, dtype=np.uint8))
    z, best, hist = local_search(f, start, budget, np.random.default_rng(seed), allowed=allowed,
                                 max_skip=max_skip)
    dec.set_skip(z)
    return z, best, hist, f0
