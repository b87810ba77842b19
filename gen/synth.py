"""Counter-based synthetic data for matrix-factorisation SGD (paper Sec. 3.1, Sec. 5).

Every random draw is a pure function of (seed, stream, index), so any slice of
a dataset can be regenerated on its own, in any order and on any number of
threads, with identical results.  The counter generator is SplitMix64
(Steele, Lea and Flood, "Fast splittable pseudorandom number generators",
OOPSLA 2014): output number n of a SplitMix64 sequence whose state starts at
s0 is mix64(s0 + n * GOLDEN).

Shapes and distributions follow the workloads of the paper's MF experiment
(Sec. 5: a Netflix-shaped 480k x 18k matrix with 100M observed entries, rank
100) with synthetic values; no record of any real dataset is used.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass

import numpy as np

GOLDEN = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB

# Stream identifiers of the input generator.
STREAM_USER = 1
STREAM_ITEM = 2
STREAM_NOISE_A = 3
STREAM_NOISE_B = 4
STREAM_TRUTH_U = 5
STREAM_TRUTH_V = 6
STREAM_INIT_L = 7
STREAM_INIT_R = 8
STREAM_PERM_USER = 9
STREAM_PERM_ITEM = 10
STREAM_SHARD = 11
STREAM_MINIBATCH = 12

_CHUNK = 1 << 21


def mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function on a uint64 array (wrapping arithmetic)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * np.uint64(_M1)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(_M2)
    return z ^ (z >> np.uint64(31))


def _stream_state(seed: int, stream: int) -> np.uint64:
    s = mix64(np.array([seed & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64))[0]
    t = mix64(np.array([stream], dtype=np.uint64))[0]
    return np.uint64(int(s) ^ int(t))


def ctr_u64(seed: int, stream: int, index) -> np.ndarray:
    """Draw number `index` (0-based) of stream `stream` under `seed`."""
    idx = np.asarray(index, dtype=np.uint64)
    s0 = _stream_state(seed, stream)
    with np.errstate(over="ignore"):
        return mix64(s0 + (idx + np.uint64(1)) * np.uint64(GOLDEN))


def _below(h: np.ndarray, n: int) -> np.ndarray:
    """Map 64-bit draws to [0, n) by the multiply-high of the top 32 bits."""
    assert 0 < n < (1 << 32)
    return ((h >> np.uint64(32)) * np.uint64(n)) >> np.uint64(32)


def _unit_open(h: np.ndarray) -> np.ndarray:
    """Map 64-bit draws to doubles in the open interval (0, 1)."""
    return ((h >> np.uint64(11)).astype(np.float64) + 0.5) * (1.0 / 9007199254740992.0)


def _normal(seed: int, stream_a: int, stream_b: int, lo: int, hi: int) -> np.ndarray:
    """Standard normals for draw indices [lo, hi) by the Box-Muller transform."""
    idx = np.arange(lo, hi, dtype=np.uint64)
    u1 = _unit_open(ctr_u64(seed, stream_a, idx))
    u2 = _unit_open(ctr_u64(seed, stream_b, idx))
    return np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * math.pi * u2)


def _threads() -> int:
    return max(1, min(16, os.cpu_count() or 1))


def _parallel(n: int, fn, chunk: int = _CHUNK) -> None:
    spans = [(lo, min(n, lo + chunk)) for lo in range(0, n, chunk)]
    if len(spans) <= 1:
        for lo, hi in spans:
            fn(lo, hi)
        return
    with ThreadPoolExecutor(_threads()) as ex:
        list(ex.map(lambda s: fn(*s), spans))


def gaussian_matrix(seed: int, stream: int, rows: int, cols: int, std: float) -> np.ndarray:
    """rows x cols float32 matrix of N(0, std^2) draws, element index r*cols+q."""
    out = np.empty(rows * cols, dtype=np.float32)

    def fill(lo, hi):
        out[lo:hi] = (std * _normal(seed, stream, stream + 100, lo, hi)).astype(np.float32)

    _parallel(rows * cols, fill)
    return out.reshape(rows, cols)


class _Zipf:
    """Zipf(a) over n ids: P(rank k) proportional to k^-a, ranks mapped to ids
    through a seeded permutation so that popular ids are scattered."""

    def __init__(self, n: int, a: float, seed: int, perm_stream: int):
        w = np.arange(1, n + 1, dtype=np.float64) ** (-a)
        cdf = np.cumsum(w)
        self.cdf = cdf / cdf[-1]
        self.cdf[-1] = 1.0
        keys = ctr_u64(seed, perm_stream, np.arange(n, dtype=np.uint64))
        self.perm = np.argsort(keys, kind="stable").astype(np.int32)
        self.n = n

    def sample(self, u: np.ndarray) -> np.ndarray:
        rank = np.searchsorted(self.cdf, u, side="right")
        np.minimum(rank, self.n - 1, out=rank)
        return self.perm[rank]


@dataclass
class MFData:
    """Observed entries D_obs of an N x M matrix plus initial factors.

    i, j: int32 user / item index of each observed entry; D: float32 value;
    L0: N x K float32 initial user factors; R0: M x K float32 initial item
    factors (stored row-major per item, i.e. the transpose of the paper's R).
    """

    n_users: int
    n_items: int
    K: int
    i: np.ndarray
    j: np.ndarray
    D: np.ndarray
    L0: np.ndarray
    R0: np.ndarray

    @property
    def n_obs(self) -> int:
        return int(self.i.shape[0])


def make_ratings(
    *,
    n_users: int,
    n_items: int,
    n_obs: int,
    seed: int,
    user_dist: str = "uniform",
    user_a: float = 1.0,
    item_dist: str = "uniform",
    item_a: float = 1.0,
    truth_rank: int = 16,
    truth_var: float = 0.25,
    noise_var: float = 0.1,
    offset: float = 0.0,
    integer_1_5: bool = False,
):
    """Observed (i, j, D): i.i.d. (i, j) pairs (duplicates allowed) and
    D = offset + U_i . V_j + N(0, noise_var), optionally rounded half away from
    zero and clipped to the integers 1..5."""
    U = gaussian_matrix(seed, STREAM_TRUTH_U, n_users, truth_rank, math.sqrt(truth_var))
    V = gaussian_matrix(seed, STREAM_TRUTH_V, n_items, truth_rank, math.sqrt(truth_var))
    zu = _Zipf(n_users, user_a, seed, STREAM_PERM_USER) if user_dist == "zipf" else None
    zi = _Zipf(n_items, item_a, seed, STREAM_PERM_ITEM) if item_dist == "zipf" else None
    I = np.empty(n_obs, dtype=np.int32)
    J = np.empty(n_obs, dtype=np.int32)
    D = np.empty(n_obs, dtype=np.float32)
    noise_std = math.sqrt(noise_var)

    def fill(lo, hi):
        idx = np.arange(lo, hi, dtype=np.uint64)
        hu = ctr_u64(seed, STREAM_USER, idx)
        hi_ = ctr_u64(seed, STREAM_ITEM, idx)
        iu = zu.sample(_unit_open(hu)) if zu is not None else _below(hu, n_users).astype(np.int32)
        ji = zi.sample(_unit_open(hi_)) if zi is not None else _below(hi_, n_items).astype(np.int32)
        dot = np.einsum("ij,ij->i", U[iu].astype(np.float64), V[ji].astype(np.float64))
        val = offset + dot + noise_std * _normal(seed, STREAM_NOISE_A, STREAM_NOISE_B, lo, hi)
        if integer_1_5:
            val = np.clip(np.sign(val) * np.floor(np.abs(val) + 0.5), 1.0, 5.0)
        I[lo:hi] = iu
        J[lo:hi] = ji
        D[lo:hi] = val.astype(np.float32)

    _parallel(n_obs, fill)
    return I, J, D


def make_mf_data(
    *,
    n_users: int,
    n_items: int,
    n_obs: int,
    K: int,
    seed: int,
    init_var: float = 0.01,
    **rating_kw,
) -> MFData:
    I, J, D = make_ratings(n_users=n_users, n_items=n_items, n_obs=n_obs, seed=seed, **rating_kw)
    std = math.sqrt(init_var)
    L0 = gaussian_matrix(seed, STREAM_INIT_L, n_users, K, std)
    R0 = gaussian_matrix(seed, STREAM_INIT_R, n_items, K, std)
    return MFData(n_users, n_items, K, I, J, D, L0, R0)


def shard_users(n_users: int, P: int, seed: int) -> np.ndarray:
    """Data partition across P workers by a seeded hash of the user index
    (Sec. 3.1: D_obs is partitioned over the worker nodes).  int32[n_users]."""
    out = np.empty(n_users, dtype=np.int32)

    def fill(lo, hi):
        h = ctr_u64(seed, STREAM_SHARD, np.arange(lo, hi, dtype=np.uint64))
        out[lo:hi] = _below(h, P).astype(np.int32)

    _parallel(n_users, fill)
    return out


def minibatch_labels(n_obs: int, F: int, seed: int) -> np.ndarray:
    """Minibatch label b(k) in [0, F) of each observed entry (Sec. 5: each
    Clock() processes a fixed fraction 1/F of the data).  uint8[n_obs]."""
    assert 1 <= F <= 255
    out = np.empty(n_obs, dtype=np.uint8)

    def fill(lo, hi):
        h = ctr_u64(seed, STREAM_MINIBATCH, np.arange(lo, hi, dtype=np.uint64))
        out[lo:hi] = _below(h, F).astype(np.uint8)

    _parallel(n_obs, fill)
    return out
