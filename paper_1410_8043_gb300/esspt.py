"""Python binding of the esspt C-ABI (argument marshalling only).

Every method maps to one `esspt_*` entry point of include/esspt.h.  PyTorch
provides device memory (the workspaces are torch tensors) and the CUDA
stream; every computation runs in the library's CUDA kernels.  There is no
CPU fallback: if the library or a GPU is missing, construction fails.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libesspt.so")

OK, EINVAL, ESTATE, ENOSPC, ESTALE, ECUDA = range(6)
STATUS_NAMES = {OK: "OK", EINVAL: "EINVAL", ESTATE: "ESTATE", ENOSPC: "ENOSPC", ESTALE: "ESTALE", ECUDA: "ECUDA"}
MODELS = {"ssp": 0, "essp": 1, "external": 2, "vap": 3, "ssp_row": 4}

# Every entry point declared in include/esspt.h.
EXPORTS = (
    "esspt_workspace_bytes", "esspt_create", "esspt_destroy", "esspt_table_init", "esspt_get", "esspt_inc",
    "esspt_clock", "esspt_set_schedule", "esspt_poll", "esspt_read_schedule", "esspt_read_table",
    "esspt_last_error", "esspt_mf_workspace_bytes", "esspt_mf_scratch_bytes", "esspt_mf_load",
    "esspt_mf_sgd_clock", "esspt_mf_objective", "esspt_mf_minibatch_size", "esspt_mf_export_minibatch",
    "esspt_mf_stage_minibatch", "esspt_mf_stage_bytes", "esspt_set_profile_events",
    "esspt_mf_worker_objective_noalloc",
    "esspt_mf_sequential_work_bytes", "esspt_mf_sgd_clock_sequential",
)


class EssptError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [
        ("n_rows", ctypes.c_int64),
        ("row_width", ctypes.c_int32),
        ("num_workers", ctypes.c_int32),
        ("staleness", ctypes.c_int32),
        ("model", ctypes.c_int32),
        ("phased", ctypes.c_int32),
        ("essp_max_delay", ctypes.c_int32),
        ("essp_p", ctypes.c_double),
        ("seed", ctypes.c_uint64),
        ("stream", ctypes.c_void_p),
        ("vap_v0", ctypes.c_double),
    ]


_lib = None


def lib() -> ctypes.CDLL:
    """Load libesspt.so (built by `build()`); raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"esspt CUDA library not built: {LIB_PATH} is missing (run __graft_entry__.build())")
    L = ctypes.CDLL(LIB_PATH)
    P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    sig = {
        "esspt_workspace_bytes": (SZ, [P]),
        "esspt_create": (ctypes.c_int, [P, P, SZ, P]),
        "esspt_destroy": (ctypes.c_int, [P]),
        "esspt_table_init": (ctypes.c_int, [P, P]),
        "esspt_get": (ctypes.c_int, [P, I32, P, I64, P, P]),
        "esspt_inc": (ctypes.c_int, [P, I32, P, P, I64]),
        "esspt_clock": (ctypes.c_int, [P]),
        "esspt_set_schedule": (ctypes.c_int, [P, P]),
        "esspt_poll": (ctypes.c_int, [P]),
        "esspt_read_schedule": (ctypes.c_int, [P, P, P]),
        "esspt_read_table": (ctypes.c_int, [P, I32, P]),
        "esspt_last_error": (ctypes.c_char_p, [P]),
        "esspt_mf_workspace_bytes": (SZ, [P, I64, I64, I32]),
        "esspt_mf_scratch_bytes": (SZ, [P, I64, I64, I32]),
        "esspt_mf_load": (ctypes.c_int, [P, P, P, P, P, I64, P, I64, I32, P, SZ, P, SZ]),
        "esspt_mf_sgd_clock": (ctypes.c_int, [P, ctypes.c_float, ctypes.c_float, I32, P]),
        "esspt_mf_sequential_work_bytes": (SZ, [P]),
        "esspt_mf_sgd_clock_sequential": (ctypes.c_int, [P, ctypes.c_float, ctypes.c_float, I32, P, P, SZ]),
        "esspt_mf_objective": (ctypes.c_int, [P, I32, ctypes.c_float, P, P, P]),
        "esspt_mf_minibatch_size": (ctypes.c_int, [P, I32, P]),
        "esspt_mf_export_minibatch": (ctypes.c_int, [P, I32, P, P, P, P]),
        "esspt_mf_stage_bytes": (SZ, [P]),
        "esspt_mf_stage_minibatch": (ctypes.c_int, [P, I32, P, P, P, P, P, SZ, P]),
        "esspt_set_profile_events": (ctypes.c_int, [P, P, P]),
        "esspt_mf_worker_objective_noalloc": (ctypes.c_int, [P, I32, ctypes.c_float, P, P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib = L
    return L


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        return t.data_ptr()
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return int(t)


def _dev_tensor(x, dtype, device) -> torch.Tensor:
    if isinstance(x, torch.Tensor):
        return x.to(device=device, dtype=dtype).contiguous()
    return torch.as_tensor(np.ascontiguousarray(x), dtype=dtype, device=device)


class Table:
    """A stale-synchronous parameter table on one GPU (one `esspt_ctx`)."""

    def __init__(self, n_rows: int, K: int, P: int, s: int, model: str = "ssp", phased: bool = True,
                 seed: int = 8043, essp_p: float = 0.7, essp_max_delay: int = 3, vap_v0: float = 0.0,
                 device=None, stream=None):
        if not torch.cuda.is_available():
            raise RuntimeError("esspt needs a CUDA device")
        L = lib()
        self.device = torch.device(device if device is not None else "cuda")
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        self.cfg = Config(n_rows, K, P, s, MODELS[model], int(phased), essp_max_delay, essp_p,
                          seed & 0xFFFFFFFFFFFFFFFF, ctypes.c_void_p(self.stream.cuda_stream), vap_v0)
        self.n_rows, self.K, self.P, self.s, self.model = n_rows, K, P, s, model
        nbytes = L.esspt_workspace_bytes(ctypes.byref(self.cfg))
        if nbytes == 0:
            raise EssptError(EINVAL, "invalid table configuration")
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        h = ctypes.c_void_p()
        st = L.esspt_create(ctypes.byref(self.cfg), self.workspace.data_ptr(), nbytes, ctypes.byref(h))
        if st != OK:
            raise EssptError(st, L.esspt_last_error(None).decode())
        self._h = h
        self.mf_workspace = None
        self.n_users = None

    # -- plumbing -----------------------------------------------------------
    def _check(self, st: int) -> None:
        if st != OK:
            raise EssptError(st, lib().esspt_last_error(self._h).decode())

    def close(self) -> None:
        if getattr(self, "_h", None):
            lib().esspt_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- table API ----------------------------------------------------------
    def table_init(self, rows) -> None:
        """esspt_table_init: version 0 from (n_rows, K) fp32 values."""
        t = _dev_tensor(rows, torch.float32, self.device)
        assert t.numel() == self.n_rows * self.K
        self._check(lib().esspt_table_init(self._h, t.data_ptr()))
        self._keep = t

    def get(self, worker: int, row_ids, out=None, want_version: bool = False):
        """esspt_get: rows of `worker`'s read version; returns (rows, version or None)."""
        ids = _dev_tensor(row_ids, torch.int32, self.device)
        if out is None:
            out = torch.empty((ids.numel(), self.K), dtype=torch.float32, device=self.device)
        ver = ctypes.c_int32(-1)
        self._check(lib().esspt_get(self._h, worker, ids.data_ptr(), ids.numel(), out.data_ptr(),
                                    ctypes.byref(ver) if want_version else None))
        self._keep_ids = ids
        return out, (ver.value if want_version else None)

    def inc(self, worker: int, row_ids, deltas) -> None:
        """esspt_inc: additive updates into the version being written."""
        ids = _dev_tensor(row_ids, torch.int32, self.device)
        d = _dev_tensor(deltas, torch.float32, self.device)
        assert d.numel() == ids.numel() * self.K
        self._check(lib().esspt_inc(self._h, worker, ids.data_ptr(), d.data_ptr(), ids.numel()))
        self._keep_inc = (ids, d)

    def clock(self) -> None:
        """esspt_clock: all workers tick."""
        self._check(lib().esspt_clock(self._h))

    def set_schedule(self, v) -> None:
        """esspt_set_schedule (external model)."""
        a = np.ascontiguousarray(v, dtype=np.int32)
        assert a.shape == (self.P,)
        self._check(lib().esspt_set_schedule(self._h, a.ctypes.data))

    def poll(self) -> None:
        """esspt_poll: synchronise and raise on a latched device error."""
        self._check(lib().esspt_poll(self._h))

    def read_schedule(self):
        """esspt_read_schedule: (v_p(c) as int32[P], c)."""
        v = np.empty(self.P, dtype=np.int32)
        c = ctypes.c_int32()
        self._check(lib().esspt_read_schedule(self._h, v.ctypes.data, ctypes.byref(c)))
        return v, c.value

    @property
    def clock_index(self) -> int:
        c = ctypes.c_int32()
        self._check(lib().esspt_read_schedule(self._h, None, ctypes.byref(c)))
        return c.value

    def read_table(self, version: int, out=None) -> torch.Tensor:
        """esspt_read_table: a final version still in the ring."""
        if out is None:
            out = torch.empty((self.n_rows, self.K), dtype=torch.float32, device=self.device)
        self._check(lib().esspt_read_table(self._h, version, out.data_ptr()))
        return out

    # -- matrix factorisation -----------------------------------------------
    def mf_load(self, i, j, D, minibatch, worker, n_users: int, F: int) -> None:
        """esspt_mf_load: observed entries and their worker / minibatch partition."""
        L = lib()
        di = _dev_tensor(i, torch.int32, self.device)
        dj = _dev_tensor(j, torch.int32, self.device)
        dD = _dev_tensor(D, torch.float32, self.device)
        dm = _dev_tensor(minibatch, torch.uint8, self.device)
        dw = _dev_tensor(worker, torch.int32, self.device)
        n_obs = di.numel()
        ws = L.esspt_mf_workspace_bytes(self._h, n_obs, n_users, F)
        sc = L.esspt_mf_scratch_bytes(self._h, n_obs, n_users, F)
        if ws == 0 or sc == 0:
            raise EssptError(EINVAL, "invalid MF sizes")
        self.mf_workspace = torch.empty(ws, dtype=torch.uint8, device=self.device)
        scratch = torch.empty(sc, dtype=torch.uint8, device=self.device)
        self._check(L.esspt_mf_load(self._h, di.data_ptr(), dj.data_ptr(), dD.data_ptr(), dm.data_ptr(), n_obs,
                                    dw.data_ptr(), n_users, F, self.mf_workspace.data_ptr(), ws,
                                    scratch.data_ptr(), sc))
        del scratch, di, dj, dD, dm, dw
        # the sort scratch and the input copies can be tens of GB: hand them back
        torch.cuda.empty_cache()
        self.n_users, self.F, self.n_obs = n_users, F, n_obs
        self._obj_scratch = torch.zeros(2, dtype=torch.float64, device=self.device)

    def mf_sgd_clock(self, eta: float, lam: float, cap: int = 0, sq_loss: torch.Tensor | None = None) -> None:
        """esspt_mf_sgd_clock: one fused clock of MF-SGD (+ CLOCK)."""
        self._check(lib().esspt_mf_sgd_clock(self._h, eta, lam, cap, _ptr(sq_loss)))

    def mf_sgd_clock_sequential(self, eta: float, lam: float, cap: int = 0,
                                sq_loss: torch.Tensor | None = None) -> None:
        """esspt_mf_sgd_clock_sequential: one clock with read-my-writes SGD inside each worker.
        The work buffer is allocated here (torch) on first use and kept."""
        need = lib().esspt_mf_sequential_work_bytes(self._h)
        if getattr(self, "_seq_work", None) is None or self._seq_work.numel() < need:
            self._seq_work = torch.empty(max(need, 16), dtype=torch.uint8, device=self.device)
        self._check(lib().esspt_mf_sgd_clock_sequential(self._h, eta, lam, cap, _ptr(sq_loss),
                                                        self._seq_work.data_ptr(), self._seq_work.numel()))

    def mf_objective(self, version: int, lam: float):
        """esspt_mf_objective: (sum e^2, sum [e^2 + lam(|L_i|^2+|R_j|^2)]) at `version`."""
        sq = ctypes.c_double()
        pen = ctypes.c_double()
        self._check(lib().esspt_mf_objective(self._h, version, lam, self._obj_scratch.data_ptr(), ctypes.byref(sq),
                                             ctypes.byref(pen)))
        return sq.value, pen.value

    def mf_minibatch_size(self, b: int) -> int:
        """esspt_mf_minibatch_size."""
        n = ctypes.c_int64()
        self._check(lib().esspt_mf_minibatch_size(self._h, b, ctypes.byref(n)))
        return n.value

    def mf_export_minibatch(self, b: int, pin: bool = True, out=None):
        """esspt_mf_export_minibatch: (u, j, D, uoff) host tensors of minibatch b,
        written into `out` (four contiguous host tensors of the right sizes) if given."""
        n = self.mf_minibatch_size(b)
        if out is not None:
            u, j, D, uoff = out
            assert u.numel() == n and j.numel() == n and D.numel() == n and uoff.numel() == self.n_users + 1
            assert u.dtype == j.dtype == uoff.dtype == torch.int32 and D.dtype == torch.float32
            assert all(x.is_contiguous() and x.device.type == "cpu" for x in out)
        else:
            mk = lambda k, dt: torch.empty(k, dtype=dt, pin_memory=pin)  # noqa: E731
            u, j, D, uoff = mk(n, torch.int32), mk(n, torch.int32), mk(n, torch.float32), mk(self.n_users + 1, torch.int32)
        self._check(lib().esspt_mf_export_minibatch(self._h, b, u.data_ptr(), j.data_ptr(), D.data_ptr(),
                                                    uoff.data_ptr()))
        return u, j, D, uoff

    def mf_stage_minibatch(self, b: int, u, j, D, uoff, stream=None) -> None:
        """esspt_mf_stage_minibatch: asynchronous host-to-device copy of minibatch b
        on `stream` (a torch.cuda.Stream; None = the table's stream).  The device
        staging buffer is allocated here (torch) on first use and kept."""
        need = lib().esspt_mf_stage_bytes(self._h)
        if getattr(self, "_stage", None) is None or self._stage.numel() < need:
            self._stage = torch.empty(max(need, 256), dtype=torch.uint8, device=self.device)
        st = None if stream is None else ctypes.c_void_p(stream.cuda_stream)
        self._check(lib().esspt_mf_stage_minibatch(self._h, b, u.data_ptr(), j.data_ptr(), D.data_ptr(),
                                                   uoff.data_ptr(), self._stage.data_ptr(), self._stage.numel(), st))

    def set_profile_events(self, before, after) -> None:
        """esspt_set_profile_events: torch.cuda.Event pair (created) or None."""
        if before is None:
            self._check(lib().esspt_set_profile_events(self._h, None, None))
        else:
            self._check(lib().esspt_set_profile_events(self._h, before.cuda_event, after.cuda_event))

    def mf_worker_objective_noalloc(self, version: int, lam: float):
        """esspt_mf_worker_objective_noalloc: per-worker (sum e^2, penalised sum)
        as two float64[P] arrays, computed without any device allocation."""
        sq = np.empty(self.P, dtype=np.float64)
        pen = np.empty(self.P, dtype=np.float64)
        self._check(lib().esspt_mf_worker_objective_noalloc(self._h, version, lam, sq.ctypes.data, pen.ctypes.data))
        return sq, pen

    @classmethod
    def for_workload(cls, w, data, partition, **kw) -> "Table":
        """A table for an MF workload (gen.workloads.Workload) with data loaded."""
        t = cls(w.n_users + w.n_items, w.K, w.P, w.s, model=w.model, seed=w.sched_seed, essp_p=w.essp_p,
                essp_max_delay=w.essp_max_delay, vap_v0=w.vap_v0, **kw)
        wp, mb = partition
        t.mf_load(data.i, data.j, data.D, mb, wp, w.n_users, w.F)
        t.table_init(np.concatenate([data.L0, data.R0]))
        return t
