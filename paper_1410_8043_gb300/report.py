"""Staleness and convergence report of the consistency models on one GPU.

For each workload it runs the clocks on the GPU through the C-ABI and
records, per clock:
  * the clock differential v_p(c) - c of every worker's read (Fig. 1 left:
    BSP always gives -1, SSP spreads reads over -1..-(s+1), ESSP keeps most
    at -1);
  * the squared loss and the penalised objective at version c (Sec. 5 plots
    the objective against clocks);
  * the device time of the clock (CUDA events on the library's stream).

    python -m paper_1410_8043_gb300.report --workloads mid,mid_essp,mid_vap --clocks 40 --out report.json

The output is one JSON object per workload, one line each.  The objective
passes are not part of the timed clock.
"""
from __future__ import annotations

import argparse
import json
import sys

import numpy as np


def run_workload(name, clocks: int | None = None) -> dict:
    """The report of one workload, given by name or as a gen.workloads.Workload."""
    import torch

    from gen import workload

    from . import esspt

    w = workload(name) if isinstance(name, str) else name
    name = w.name
    C = w.clocks if clocks is None else clocks
    d = w.make_data()
    part = w.partition()
    dev = torch.device("cuda")
    stream = torch.cuda.Stream(dev)
    with torch.cuda.stream(stream):
        t = esspt.Table.for_workload(w, d, part, device=dev, stream=stream)
    mb = part[1]
    per_clock = []
    hist_all = np.zeros(w.s + 1, np.int64)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sq0, pen0 = t.mf_objective(0, w.lam)
    for c in range(1, C + 1):
        v, clk = t.read_schedule()
        assert clk == c
        hist = np.bincount(c - 1 - v, minlength=w.s + 1)[: w.s + 1]
        hist_all += hist
        e0.record(stream)
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        sq, pen = t.mf_objective(c, w.lam)
        per_clock.append({
            "clock": c,
            "ms": e0.elapsed_time(e1),
            "ratings": int(np.count_nonzero(mb == (c - 1) % w.F)),
            "sq_loss": sq,
            "penalised": pen,
            "clock_differential": {str(-1 - k): int(hist[k]) for k in range(w.s + 1)},
        })
    t.poll()
    t.close()
    # The first clocks warm the kernels; the throughput skips them.
    warm = per_clock[3:] if len(per_clock) > 6 else per_clock
    ms = float(np.median([r["ms"] for r in warm]))
    n = float(np.mean([r["ratings"] for r in warm]))
    return {
        "workload": name,
        "model": w.model,
        "s": w.s,
        "P": w.P,
        "vap_v0": w.vap_v0 if w.model == "vap" else None,
        "clocks": C,
        "objective_at_0": {"sq_loss": sq0, "penalised": pen0},
        "median_ms_per_clock": ms,
        "ratings_per_s": n / (ms / 1e3),
        "clock_differential": {str(-1 - k): float(hist_all[k] / hist_all.sum()) for k in range(w.s + 1)},
        "mean_staleness": float(np.dot(np.arange(w.s + 1), hist_all) / hist_all.sum()),
        "per_clock": per_clock,
    }


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workloads", default="mid,mid_essp,mid_vap")
    ap.add_argument("--clocks", type=int, default=None, help="clocks per workload (default: the workload's)")
    ap.add_argument("--out", default="-", help="output file, - for stdout")
    args = ap.parse_args(argv)
    out = sys.stdout if args.out == "-" else open(args.out, "w")
    for name in args.workloads.split(","):
        out.write(json.dumps(run_workload(name.strip(), args.clocks)) + "\n")
        out.flush()
    if out is not sys.stdout:
        out.close()
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
