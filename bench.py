"""Benchmark: stale-synchronous MF-SGD clocks on GB300 (ratings per second).

One step = one whole clock of the hot path (read-version schedule, fused SGD
gather/residual/update with the user-row merge, the Clock() merge of the
item rows) over one minibatch.  The headline workload is the large one
(10M x 1M, 2B entries, Zipf(1.1) users and items, rank 64, 128 workers,
SSP s=4, 1/50 of the data per clock); the Netflix-shaped mid workload
(480k x 18k, 100M entries, rank 100, 32 workers, SSP s=3, 1/20 per clock)
is measured in the same run and reported under "extra_workloads".

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload large] [--extra mid]
    python bench.py --impl reference ...   # the fp64 CPU oracle, same metric

Prints one JSON line.  With N > 1 (torchrun) every rank runs an independent
replica of the workload on its own GPU: the method has no cross-GPU step.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "SGD ratings/sec per clock on 1 GB300; achieved HBM GB/s vs peak"
UNIT = "ratings/s"


def kernel_code_digest(text: str) -> str:
    """First 16 hex digits of the SHA-256 of a CUDA source's code: comments
    removed and every run of whitespace made one space, so that editing a
    comment keeps the digest and any change to the code changes it."""
    import hashlib
    import re

    code = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    code = re.sub(r"//[^\n]*", " ", code)
    code = " ".join(code.split())
    return hashlib.sha256(code.encode()).hexdigest()[:16]


def _profiled_traffic(kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` on `workload` from its committed ncu
    summary profiles/<kernel>_<workload>.md, or None when there is none or the
    kernels' code changed since the capture."""
    src = os.path.join(ROOT, "paper_1410_8043_gb300", "csrc", "mf_kernels.cu")
    try:
        digest = kernel_code_digest(open(src).read())
    except OSError:
        return None
    for path in [os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")]:
        if not os.path.exists(path):
            continue
        fields = {}
        for line in open(path):
            if ":" in line and not line.startswith(("|", "#", " ", "`")):
                k, _, v = line.partition(":")
                fields[k.strip()] = v.strip()
        if fields.get("kernel_code_sha256_16") == digest and "traffic_bytes_per_launch" in fields:
            return float(fields["traffic_bytes_per_launch"])
    return None


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi SM clock / throttle-reason samples while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.rows = []
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append((time.time(), line.strip()))

    def mark(self, which):
        setattr(self, which, time.time())

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.15)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        rows = [r for t, r in self.rows if self.t0 is None or (self.t0 - 0.1 <= t <= (self.t1 or t) + 0.1)]
        if not rows:
            rows = [r for _, r in self.rows]
        for r in rows:
            f = [x.strip() for x in r.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, val in zip(names, f[4:8]):
                if val.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def _barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def _reduce_over_ranks(world, x: float, op: str) -> float:
    """Max or sum of a host scalar over the ranks (NCCL on GPUs, gloo on CPU)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def _max_over_ranks(world, x: float) -> float:
    return _reduce_over_ranks(world, x, "max")


def _sum_over_ranks(world, x: float) -> float:
    return _reduce_over_ranks(world, x, "sum")


def replica_throughput(world, ratings: float, ms: float) -> float:
    """Whole-job ratings/s of N independent replicas: all ratings over the slowest rank's time."""
    return _sum_over_ranks(world, ratings) / (_max_over_ranks(world, ms) / 1e3)


class FloorModel:
    """Compulsory HBM bytes of the SGD kernels of one clock (minibatch b, read
    versions v): 12 B per entry (i, j, D); the merge of every user row (read
    version c-1, write version c); each user row read at a stale version
    (v != c-1) by a user with entries; each distinct (item, stale version)
    row read.  Item rows of version c-1 count as resident (the previous
    clock's merge just wrote them).  Counted with torch on `device` (the
    distinct pairs by sorting), one minibatch at a time.

    On the work-list path (32 < K <= 64) an idle user row unchanged over the
    last s+2 clocks is not merged (its ring slot already holds it), and each
    user has a 4-byte change-clock word, read for idle users and written for
    active ones.  `bytes` must then see every clock from the table's version
    0 in order."""

    def __init__(self, w, data, wp, mb, device="cpu"):
        import torch

        self.w = w
        self.dev = torch.device(device)
        self.i = torch.as_tensor(np.ascontiguousarray(data.i)).to(self.dev)
        self.j = torch.as_tensor(np.ascontiguousarray(data.j)).to(self.dev)
        self.mb = torch.as_tensor(np.ascontiguousarray(mb)).to(self.dev)
        self.wp = torch.as_tensor(np.ascontiguousarray(wp)).to(self.dev).long()
        self._b = None
        self._per_b = {}
        self.skip = 32 < w.K <= 64
        self.chg = torch.zeros(w.n_users, dtype=torch.int64, device=self.dev) if self.skip else None
        self.last_c = 0

    def _minibatch(self, b):
        """(entries, worker of each user with entries, distinct worker*M + item
        pairs, some user has more than 96 entries) of minibatch b."""
        import torch

        if self._b != b:
            idx = torch.nonzero(self.mb == b).squeeze(1)
            ui = self.i[idx].long()
            jj = self.j[idx].long()
            users, cnt = torch.unique(ui, return_counts=True)
            uw = self.wp[users]
            pj = torch.unique(self.wp[ui] * self.w.n_items + jj)
            heavy = bool(cnt.numel() and int(cnt.max()) > 96)
            self._cache = (int(idx.numel()), uw, pj, heavy, users)
            self._b = b
            del idx, ui, jj, users, cnt
        return self._cache

    def heavy(self, b) -> bool:
        """Whether minibatch b has a user with more than 96 entries (those go
        through the chunk and heavy-merge kernels)."""
        if b not in self._per_b:
            self._per_b[b] = self._minibatch(b)[3]
        return self._per_b[b]

    def bytes(self, c, v):
        import torch

        w = self.w
        b = (c - 1) % w.F
        n, uw, pj, heavy, active = self._minibatch(b)
        self._per_b[b] = heavy
        vt = torch.as_tensor(np.ascontiguousarray(v, dtype=np.int64)).to(self.dev)
        stale = vt != (c - 1)
        users = int(stale[uw].sum())
        p = pj // w.n_items
        sp = stale[p]
        items = int(torch.unique(vt[p[sp]] * w.n_items + (pj[sp] % w.n_items)).numel())
        merged = w.n_users
        words = 0
        if self.skip:
            assert c == self.last_c + 1, "the work-list floor needs every clock in order"
            self.last_c = c
            idle = torch.ones(w.n_users, dtype=torch.bool, device=self.dev)
            idle[active] = False
            skipped = int((idle & (c - self.chg >= w.s + 2)).sum())
            merged = w.n_users - skipped
            words = 4 * w.n_users
            self.chg[active] = c
        return 12 * n + 8 * w.K * merged + words + 4 * w.K * (users + items), n


def _model_launches(w, c):
    """Kernels the read model adds to clock c: VAP's norms for clock c+1 (one
    per 8 candidate versions) and its schedule; the row-granular cache's
    refresh before the SGD kernels."""
    if w.model == "vap":
        return (min(w.s, c) + 7) // 8 + 1
    if w.model == "ssp_row":
        return 1
    return 0


def _stage_overlapped(t, w, host_mb, W, K, stream, copy_stream, loss_d, loss_h):
    """K clocks through the public API with host inputs: minibatch of clock
    c+1 is copied from pinned host memory on `copy_stream` while clock c runs
    on `stream`; each clock's squared loss is copied back to pinned host
    memory.  Returns (start event on `stream`, h2d bytes, d2h bytes)."""
    import torch

    F = w.F
    staged = [torch.cuda.Event() for _ in range(K)]
    done = [torch.cuda.Event() for _ in range(K)]
    h2d = d2h = 0

    def stage(k):
        nonlocal h2d
        c = W + 1 + k
        b = (c - 1) % F
        # minibatch b was last read by clock c - F: wait for it
        if k - F >= 0:
            copy_stream.wait_event(done[k - F])
        u, j, D, uoff = host_mb[b]
        t.mf_stage_minibatch(b, u, j, D, uoff, stream=copy_stream)
        staged[k].record(copy_stream)
        h2d += 4 * (u.numel() + j.numel() + D.numel() + uoff.numel())

    start = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    copy_stream.wait_event(start)
    stage(0)
    for k in range(K):
        if k + 1 < K:
            stage(k + 1)
        stream.wait_event(staged[k])
        t.mf_sgd_clock(w.eta, w.lam, w.cap, sq_loss=loss_d[k:k + 1])
        with torch.cuda.stream(stream):
            loss_h[k:k + 1].copy_(loss_d[k:k + 1], non_blocking=True)
        d2h += 8
        done[k].record(stream)
    return start, h2d, d2h


class HostBuffer:
    """One page-locked host allocation for the end-to-end minibatches.

    It is an anonymous mapping advised to use transparent huge pages and
    registered with the CUDA runtime.  The GPU reads host memory through an
    address translation on the host link, and tens of GB of small pages
    overflow it: copies from a 26 GB set of ordinary pinned buffers slowed from
    2.5 ms to 4-20 ms each.  With huge pages every copy ran at the link's
    speed.  Falls back to torch's pinned allocator if registration fails."""

    def __init__(self, n_int32: int):
        import mmap

        import torch

        self.mm = None
        nbytes = ((n_int32 * 4 + (1 << 21) - 1) >> 21) << 21
        try:
            mm = mmap.mmap(-1, nbytes, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
            if hasattr(mmap, "MADV_HUGEPAGE"):
                mm.madvise(mmap.MADV_HUGEPAGE)
            arr = np.frombuffer(mm, dtype=np.int32)
            arr[:] = 0  # fault the pages in before registering them
            if int(torch.cuda.cudart().cudaHostRegister(arr.ctypes.data, nbytes, 0)) != 0:
                raise RuntimeError("cudaHostRegister failed")
            self.mm, self.arr, self.nbytes = mm, arr, nbytes
            self.tensor = torch.from_numpy(arr[:n_int32])
            self.kind = "huge-page mapping registered with CUDA"
        except Exception:
            self.tensor = torch.empty(n_int32, dtype=torch.int32, pin_memory=True)
            self.kind = "torch pinned memory"

    def close(self):
        import torch

        if self.mm is not None:
            torch.cuda.cudart().cudaHostUnregister(self.arr.ctypes.data)
            self.tensor = self.arr = None
            try:
                self.mm.close()
            except BufferError:  # a view is still alive: the mapping goes with it
                pass
            self.mm = None


def _export_host_minibatches(t, w, need):
    """The minibatches `need` as host tensors (u, j, D, uoff), all views of one
    page-locked HostBuffer.  Returns (dict, buffer); close the buffer after
    use."""
    import torch

    sizes = {b: t.mf_minibatch_size(b) for b in need}
    buf = HostBuffer(sum(3 * n + w.n_users + 1 for n in sizes.values()))
    big = buf.tensor
    out, o = {}, 0
    for b in need:
        n = sizes[b]
        u, j, D, uoff = (big[o:o + n], big[o + n:o + 2 * n], big[o + 2 * n:o + 3 * n].view(torch.float32),
                         big[o + 3 * n:o + 3 * n + w.n_users + 1])
        o += 3 * n + w.n_users + 1
        out[b] = t.mf_export_minibatch(b, out=(u, j, D, uoff))
    return out, buf


def measure(args, w, dev, world, rank, local):
    """One workload: accounting pass, the timed clocks, the end-to-end clocks.
    Returns the bench fields of that workload, plus the data for the CPU
    baseline."""
    import torch

    from paper_1410_8043_gb300 import esspt

    t0 = time.time()
    data = w.make_data()
    wp, mb = w.partition()
    gen_s = time.time() - t0
    stream = torch.cuda.Stream(dev)
    t0 = time.time()
    with torch.cuda.stream(stream):
        t = esspt.Table.for_workload(w, data, (wp, mb), device=dev, stream=stream)
    load_s = time.time() - t0
    x0 = torch.as_tensor(np.concatenate([data.L0, data.R0]), device=dev)
    model = FloorModel(w, data, wp, mb, device=dev)

    K, W = args.steps, args.warmup
    # Accounting pass (untimed): read versions of every clock -> floor bytes.
    floors, counts = [], []
    stale = np.zeros(w.s + 1, np.int64)
    for c in range(1, W + K + 1):
        v, clk = t.read_schedule()
        assert clk == c
        fb, n = model.bytes(c, v)  # every clock: the work-list floor follows the rows' history
        if c > W:
            floors.append(fb)
            counts.append(n)
            stale += np.bincount(c - 1 - v, minlength=w.s + 1)[: w.s + 1]
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
    t.poll()
    heavy = {b: model.heavy(b) for b in {(c - 1) % w.F for c in range(W + 1, W + K + 1)}}
    del model
    torch.cuda.empty_cache()

    # Timed run from version 0 again.
    t.table_init(x0)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    for a, b_ in ev:  # create the events on the stream
        a.record(stream)
        b_.record(stream)
    for _ in range(W):
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    _barrier(world)
    torch.cuda.synchronize(dev)
    sampler.mark("t0")
    start.record(stream)
    for k in range(K):
        t.set_profile_events(ev[k][0], ev[k][1])
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
    stop.record(stream)
    torch.cuda.synchronize(dev)
    sampler.mark("t1")
    _barrier(world)
    t.set_profile_events(None, None)
    clocks = sampler.stop()
    t.poll()
    ms = start.elapsed_time(stop)
    kern_ms = [a.elapsed_time(b_) for a, b_ in ev]
    ms_max = _max_over_ranks(world, ms)
    ratings = float(sum(counts))
    total_ratings = _sum_over_ranks(world, ratings)
    value = replica_throughput(world, ratings, ms)
    c_final = t.clock_index - 1
    sq, pen = t.mf_objective(c_final, w.lam)

    # End to end through the public API: every clock's minibatch comes from
    # pinned host memory (the copy of clock c+1 overlaps clock c) and every
    # clock's squared loss goes back to the host.
    t.table_init(x0)
    need = sorted({(c - 1) % w.F for c in range(W + 1, W + K + 1)})
    host_mb, host_buf = _export_host_minibatches(t, w, need)
    copy_stream = torch.cuda.Stream(dev)
    loss_d = torch.zeros(K, dtype=torch.float64, device=dev)
    loss_h = torch.empty(K, dtype=torch.float64, pin_memory=True)
    for _ in range(W):
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
    # Untimed: stage every minibatch once.  This sizes the staging buffer and
    # pays the one-time cost of the first DMA read of freshly pinned memory
    # (about 20 ms per 0.5 GB on the GB300's host link), which a training loop
    # pays once, not per clock.
    for b in need:
        t.mf_stage_minibatch(b, *host_mb[b], stream=stream)
    torch.cuda.synchronize(dev)
    t.poll()
    _barrier(world)
    wall0 = time.time()
    e0, h2d, d2h = _stage_overlapped(t, w, host_mb, W, K, stream, copy_stream, loss_d, loss_h)
    e1 = torch.cuda.Event(enable_timing=True)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    wall = time.time() - wall0
    _barrier(world)
    e2e_ms = max(e0.elapsed_time(e1), wall * 1e3)
    e2e_ms = _max_over_ranks(world, e2e_ms)
    e2e_value = total_ratings / (e2e_ms / 1e3)
    t.poll()
    del host_mb
    host_kind = host_buf.kind
    host_buf.close()

    kern_avg_s = statistics.mean(kern_ms) / 1e3
    floor_avg = statistics.mean(floors)
    peak, peak_kind = _peaks()
    achieved = floor_avg / kern_avg_s / 1e9
    # Compulsory bytes over the measured time cannot beat the copy peak by
    # much; if they do, the floor model counts bytes the kernels never move.
    if achieved > 1.25 * peak:
        raise RuntimeError(f"floor bytes give {achieved:.0f} GB/s, above the measured peak {peak:.0f} GB/s")
    kernel = _sgd_kernel_name(w.K)
    n_avg = ratings / K
    out = {
        "value": value,
        "ms_per_step": ms_max / K,
        "config": {
            "workload": f"{w.name}: {w.n_users}x{w.n_items}, {w.n_obs} entries, rank {w.K}, P={w.P}, "
                        f"F={w.F}, {w.model.upper()} s={w.s}"
                        + (f" v0={w.vap_v0}" if w.model == "vap" else "")
                        + f", eta={w.eta}, lambda={w.lam}, cap={w.cap}",
            "parallelism": f"replicas x{world}" if world > 1 else "1 GPU",
            "l2": "inputs larger than L2 (version ring %.2f GB, entries %.2f GB; ~%.0f MB streamed per clock)"
                  % ((w.s + 2) * (w.n_users + w.n_items) * w.K * 4 / 1e9, w.n_obs * 12 / 1e9, floor_avg / 1e6),
            "ratings_per_clock": n_avg,
        },
        "roofline": {
            "bound": "hbm",
            "kernel": kernel,
            "achieved": achieved,
            "peak": peak,
            "peak_kind": peak_kind,
            "unit": "GB/s",
            "frac": achieved / peak,
            "traffic": _profiled_traffic(kernel.split(" ")[0], w.name),
            "algorithmic_bytes_per_launch": floor_avg,
            "kernel_ms": statistics.mean(kern_ms),
            # compulsory bytes per rating of the SGD launch (the figure `achieved` uses)
            "modelled_bytes_per_rating": floor_avg / n_avg,
            # an upper bound that ignores every reuse in L2: 12 + 16K + 8K(N+M)/n
            "no_reuse_bytes_per_rating": 12 + 16 * w.K + 8 * w.K * (w.n_users + w.n_items) / n_avg,
        },
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d // K, "d2h_bytes_per_step": d2h // K,
                "copies": "minibatch of clock c+1 staged on a second stream while clock c runs",
                "host_memory": host_kind},
        # per clock: the SGD kernels and the item merge (which also computes the
        # next schedule), plus the read model's own kernels
        "gpu_launches": int(sum(_sgd_launches(w.K, heavy[(c - 1) % w.F]) + _model_launches(w, c)
                                for c in range(W + 1, W + K + 1))),
        "clocks": clocks,
        "objective": {"clock": c_final, "sq_loss": sq, "penalised": pen},
        # Fig. 1 (left) quantity: clock differential v_p(c) - c of every read in
        # the timed clocks (-1 = freshest version; BSP always gives -1).
        "clock_differential": {str(-1 - k): float(stale[k] / stale.sum()) for k in range(w.s + 1)},
        "setup_s": {"generate": gen_s, "load": load_s},
    }
    t.close()
    del t, x0
    torch.cuda.empty_cache()
    return out, data, (wp, mb)


def _sgd_kernel_name(K):
    """The SGD launches of one clock that the profile events bracket."""
    if 32 < K <= 64:
        return "sgd_work16_kernel (+ user_copy_kernel, and heavy_merge_kernel when some user is heavy)"
    if 64 < K <= 128:
        return "sgd_users32_kernel (+ sgd_chunks_kernel / heavy_merge_kernel when some user is heavy)"
    return "sgd_users_kernel (+ sgd_chunks_kernel / heavy_merge_kernel when some user is heavy)"


def _sgd_launches(K, heavy: bool) -> int:
    """Kernels of one clock's SGD phase plus the item merge (which also
    computes the next schedule)."""
    if 32 < K <= 64:  # forward copy, work list, heavy merge
        return 2 + int(heavy) + 1
    return 1 + 2 * int(heavy) + 1


def run_gpu(args, w):
    import torch

    from gen import workload

    world, rank, local = _dist()
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    res, data, part = measure(args, w, dev, world, rank, local)
    out = {
        "metric": METRIC,
        "value": res.pop("value"),
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": res.pop("ms_per_step"),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic (seeded counter generator; Netflix-shaped, no real records)",
    }
    out.update(res)
    extra = [x for x in args.extra.split(",") if x and x != "none" and x != w.name]
    if extra:
        out["extra_workloads"] = {}
        for name in extra:
            r, _, _ = measure(args, workload(name), dev, world, rank, local)
            out["extra_workloads"][name] = r
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(w, data, part, clocks=args.cpu_clocks)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


def cpu_baseline(w, data, partition, clocks=2):
    """The fp64 oracle, as it stands, on the first `clocks` clocks of the same
    workload (single host thread)."""
    from oracle import Oracle

    o = Oracle.from_workload(w, data, partition)
    wp, mb = partition
    n = 0
    t0 = time.time()
    for c in range(1, clocks + 1):
        o.clock()
        n += int(np.count_nonzero(mb == (c - 1) % w.F))
    dt = time.time() - t0
    return {"value": n / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"first {clocks} clocks of {w.name} ({n} entries, full table), fp64, 1 thread",
            "seconds": dt}


def run_reference(args, w):
    """The oracle as the reference arm: each step is one oracle clock over a
    bounded sample of the workload (the entries of the first 2% of users,
    all items, same rank / workers / staleness / step size)."""
    world, rank, _ = _dist()
    if rank != 0:
        return
    from gen.synth import MFData
    from oracle import Oracle, OracleConfig

    data = w.make_data()
    wp, mb = w.partition()
    n_sub = max(1, w.n_users // 50)
    keep = data.i < n_sub
    sub = MFData(n_sub, w.n_items, w.K, data.i[keep], data.j[keep], data.D[keep], data.L0[:n_sub], data.R0)
    cfg = OracleConfig.from_workload(w, n_users=n_sub)
    o = Oracle(cfg, sub.i, sub.j, sub.D, mb[keep], wp[:n_sub], sub.L0, sub.R0)
    mbk = mb[keep]
    for _ in range(args.warmup):
        o.clock()
    n = 0
    t0 = time.time()
    for _ in range(args.steps):
        c = o.version + 1
        o.clock()
        n += int(np.count_nonzero(mbk == (c - 1) % w.F))
    dt = time.time() - t0
    sample = (f"{w.name} restricted to users [0, {n_sub}) and their {int(keep.sum())} entries, all {w.n_items} "
              f"items, one oracle clock per step, fp64, 1 thread")
    out = {
        "impl": "reference",
        "metric": METRIC,
        "value": n / dt,
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": dt * 1e3 / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": f"{w.name} (bounded sample, see cpu_baseline.sample)"},
        "cpu_baseline": {"value": n / dt, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": n / dt, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="esspt", choices=["esspt", "reference"])
    ap.add_argument("--workload", default="large")
    ap.add_argument("--extra", default="mid", help="comma-separated workloads also measured (reported under "
                    "extra_workloads), or none")
    ap.add_argument("--cpu-clocks", type=int, default=2)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    from gen import workload

    w = workload(args.workload)
    if args.impl == "reference":
        run_reference(args, w)
    else:
        run_gpu(args, w)


if __name__ == "__main__":
    main()
