"""ctypes binding of the fp64 C oracle (test infrastructure only).

The C source (esspt_oracle.c) is compiled with gcc on first use, or by
`build()`, into oracle/_lib/.  Strict IEEE arithmetic: no fast-math and no
floating-point contraction, so x86-64 and aarch64 hosts give identical bits.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "esspt_oracle.c")
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "libesspt_oracle.so")

MODELS = {"ssp": 0, "essp": 1, "external": 2, "vap": 3, "ssp_row": 4}


def build(force: bool = False) -> str:
    """Compile the oracle shared library; returns its path."""
    os.makedirs(_LIBDIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "esspt_oracle.h"))
    ):
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off",
             "-fno-fast-math", "-o", tmp, _SRC, "-lm"]
        )
        os.replace(tmp, _LIB)
    return _LIB


class _Cfg(ctypes.Structure):
    _fields_ = [
        ("n_users", ctypes.c_int64),
        ("n_items", ctypes.c_int64),
        ("K", ctypes.c_int32),
        ("P", ctypes.c_int32),
        ("s", ctypes.c_int32),
        ("F", ctypes.c_int32),
        ("model", ctypes.c_int32),
        ("phased", ctypes.c_int32),
        ("seed", ctypes.c_uint64),
        ("essp_p", ctypes.c_double),
        ("essp_max_delay", ctypes.c_int32),
        ("cap", ctypes.c_int32),
        ("eta", ctypes.c_double),
        ("lam", ctypes.c_double),
        ("keep_all", ctypes.c_int32),
        ("vap_v0", ctypes.c_double),
        ("eta_decay", ctypes.c_int32),
        ("sequential", ctypes.c_int32),
    ]


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        lib.orc_create.restype = P
        lib.orc_create.argtypes = [P, ctypes.c_int64, P, P, P, P, P, P, P]
        lib.orc_destroy.argtypes = [P]
        lib.orc_clock.argtypes = [P, P]
        lib.orc_clock.restype = ctypes.c_int
        lib.orc_version.argtypes = [P]
        lib.orc_version.restype = ctypes.c_int32
        lib.orc_schedule.argtypes = [P, P]
        lib.orc_table.argtypes = [P, ctypes.c_int32, P]
        lib.orc_objective.argtypes = [P, ctypes.c_int32, P, P]
        lib.orc_schedule_rule.argtypes = [P, ctypes.c_int32, P, P]
        lib.orc_schedule_rule.restype = ctypes.c_int
        lib.orc_ctr_u64.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64]
        lib.orc_ctr_u64.restype = ctypes.c_uint64
        lib.orc_vap_norms.argtypes = [P, P, P]
        lib.orc_vap_norms.restype = ctypes.c_int
        lib.orc_essp_thresholds.argtypes = [P, P]
        lib.orc_essp_thresholds.restype = ctypes.c_int
        lib.orc_clock_loss.argtypes = [P, P]
        lib.orc_clock_loss.restype = ctypes.c_int
        lib.orc_row_version.argtypes = [P, ctypes.c_int32, ctypes.c_int64, P]
        lib.orc_row_version.restype = ctypes.c_int
        _lib = lib
    return _lib


@dataclass
class OracleConfig:
    n_users: int
    n_items: int
    K: int
    P: int
    s: int
    F: int
    model: str = "ssp"
    phased: bool = True
    seed: int = 8043
    essp_p: float = 0.7
    essp_max_delay: int = 3
    cap: int = 0
    eta: float = 0.01
    lam: float = 0.05
    keep_all: bool = False
    vap_v0: float = 0.0
    eta_decay: bool = False
    sequential: bool = False

    def _c(self) -> _Cfg:
        return _Cfg(
            self.n_users, self.n_items, self.K, self.P, self.s, self.F, MODELS[self.model],
            int(self.phased), self.seed & 0xFFFFFFFFFFFFFFFF, self.essp_p, self.essp_max_delay,
            self.cap, self.eta, self.lam, int(self.keep_all), self.vap_v0, int(self.eta_decay),
            int(self.sequential),
        )

    @classmethod
    def from_workload(cls, w, **kw) -> "OracleConfig":
        base = dict(
            n_users=w.n_users, n_items=w.n_items, K=w.K, P=w.P, s=w.s, F=w.F, model=w.model,
            seed=w.sched_seed, essp_p=w.essp_p, essp_max_delay=w.essp_max_delay, cap=w.cap,
            eta=w.eta, lam=w.lam, vap_v0=w.vap_v0,
        )
        base.update(kw)
        return cls(**base)


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


class Oracle:
    """Stateful fp64 oracle: one `clock()` call is one Clock() of all workers."""

    def __init__(self, cfg: OracleConfig, i, j, D, minibatch, user_worker, L0, R0):
        lib = _load()
        self.cfg = cfg
        self._arrays = [
            np.ascontiguousarray(i, dtype=np.int32),
            np.ascontiguousarray(j, dtype=np.int32),
            np.ascontiguousarray(D, dtype=np.float32),
            np.ascontiguousarray(minibatch, dtype=np.uint8),
            np.ascontiguousarray(user_worker, dtype=np.int32),
            np.ascontiguousarray(L0, dtype=np.float32).reshape(cfg.n_users, cfg.K),
            np.ascontiguousarray(R0, dtype=np.float32).reshape(cfg.n_items, cfg.K),
        ]
        a = self._arrays
        n_obs = a[0].shape[0]
        assert a[1].shape[0] == n_obs and a[2].shape[0] == n_obs and a[3].shape[0] == n_obs
        assert a[4].shape[0] == cfg.n_users
        if n_obs:
            assert int(a[0].min()) >= 0 and int(a[0].max()) < cfg.n_users
            assert int(a[1].min()) >= 0 and int(a[1].max()) < cfg.n_items
            assert int(a[3].max()) < cfg.F
        assert a[4].size == 0 or (int(a[4].min()) >= 0 and int(a[4].max()) < cfg.P)
        self._ccfg = cfg._c()
        self._h = lib.orc_create(ctypes.byref(self._ccfg), n_obs, *[_ptr(x) for x in a])
        if not self._h:
            raise ValueError("oracle: invalid configuration or out of memory")
        self.rows = cfg.n_users + cfg.n_items

    @classmethod
    def from_workload(cls, w, data, partition=None, **kw) -> "Oracle":
        wp, mb = partition if partition is not None else w.partition()
        return cls(OracleConfig.from_workload(w, **kw), data.i, data.j, data.D, mb, wp, data.L0, data.R0)

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            _load().orc_destroy(h)
            self._h = None

    @property
    def version(self) -> int:
        return int(_load().orc_version(self._h))

    def clock(self, v_ext=None) -> None:
        arr = None
        if v_ext is not None:
            arr = np.ascontiguousarray(v_ext, dtype=np.int32)
            assert arr.shape[0] == self.cfg.P
        rc = _load().orc_clock(self._h, None if arr is None else _ptr(arr))
        if rc == -1:
            raise ValueError("oracle: staleness bound violated")
        if rc != 0:
            raise MemoryError("oracle: allocation failed")

    def vap_norms(self):
        """VAP: (|X[c-1] - X[c-1-k]|_inf for k = 0..s, the bound) of the last clock."""
        out = np.empty(self.cfg.s + 1, dtype=np.float64)
        b = ctypes.c_double()
        if _load().orc_vap_norms(self._h, _ptr(out), ctypes.byref(b)) != 0:
            raise ValueError("oracle: not a VAP run, or no clock has run")
        return out, b.value

    def clock_loss(self) -> float:
        """Sum of e^2 over the last clock's entries, each at its read version."""
        out = ctypes.c_double()
        if _load().orc_clock_loss(self._h, ctypes.byref(out)) != 0:
            raise ValueError("oracle: no clock has run")
        return out.value

    def row_version(self, p: int, r: int) -> int:
        """Row-granular SSP: the version worker p holds row r at (-1: never read)."""
        out = ctypes.c_int32()
        if _load().orc_row_version(self._h, p, r, ctypes.byref(out)) != 0:
            raise ValueError("oracle: not a row-granular run, or bad worker/row")
        return out.value

    def schedule(self) -> np.ndarray:
        out = np.empty(self.cfg.P, dtype=np.int32)
        if _load().orc_schedule(self._h, _ptr(out)) != 0:
            raise ValueError("oracle: no clock has run")
        return out

    def table(self, version: int | None = None) -> np.ndarray:
        v = self.version if version is None else version
        out = np.empty((self.rows, self.cfg.K), dtype=np.float64)
        if _load().orc_table(self._h, v, _ptr(out)) != 0:
            raise ValueError(f"oracle: version {v} not held")
        return out

    def objective(self, version: int | None = None):
        v = self.version if version is None else version
        sq = ctypes.c_double()
        pen = ctypes.c_double()
        if _load().orc_objective(self._h, v, ctypes.byref(sq), ctypes.byref(pen)) != 0:
            raise ValueError(f"oracle: version {v} not held")
        return sq.value, pen.value


def schedule_rule(cfg: OracleConfig, c: int, v_prev=None):
    """Read versions of clock c from the oracle's rule; None if out of bound."""
    lib = _load()
    prev = np.zeros(cfg.P, dtype=np.int32) if v_prev is None else np.ascontiguousarray(v_prev, dtype=np.int32)
    out = np.empty(cfg.P, dtype=np.int32)
    cc = cfg._c()
    rc = lib.orc_schedule_rule(ctypes.byref(cc), c, _ptr(prev), _ptr(out))
    return None if rc != 0 else out


def essp_thresholds(cfg: OracleConfig) -> list:
    """The ESSP delay thresholds floor((1-p)^k 2^32), k = 1..essp_max_delay."""
    out = np.zeros(max(1, cfg.essp_max_delay), dtype=np.uint32)
    cc = cfg._c()
    n = _load().orc_essp_thresholds(ctypes.byref(cc), _ptr(out))
    return [int(x) for x in out[:n]]


def ctr_u64(seed: int, stream: int, index: int) -> int:
    return int(_load().orc_ctr_u64(seed & 0xFFFFFFFFFFFFFFFF, stream, index))
