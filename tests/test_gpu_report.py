"""The staleness and convergence report (Fig. 1 left; Sec. 5) against the oracle.

paper_1410_8043_gb300.report runs the clocks on the GPU through the C-ABI and
records, per clock, the clock differential v_p(c) - c of every worker's read
and the objective.  Both must equal what the oracle's schedule and tables
give: the histograms exactly, the objective within 1e-5 relative (tiny).
With many workers the ESSP share of freshest reads (differential -1) must
match the closed form P(delay = 0) = 0.7 of the Geometric(0.7) push delay.
"""
import numpy as np
import pytest

from gen import workload
from oracle import Oracle

pytestmark = pytest.mark.gpu


def _oracle_report(w):
    d = w.make_data()
    o = Oracle.from_workload(w, d, w.partition())
    hist, obj = [], []
    for c in range(1, w.clocks + 1):
        o.clock()
        v = o.schedule()
        hist.append(np.bincount(c - 1 - v, minlength=w.s + 1)[: w.s + 1])
        obj.append(o.objective(c))
    return hist, obj


@pytest.mark.parametrize("model", ["ssp", "essp"])
def test_report_matches_oracle(model):
    from paper_1410_8043_gb300 import report

    w = workload("tiny").with_(name=f"tiny_{model}", model=model)
    rep = report.run_workload(w)
    hist, obj = _oracle_report(w)
    assert rep["clocks"] == w.clocks and len(rep["per_clock"]) == w.clocks
    for c, row in enumerate(rep["per_clock"], start=1):
        got = [row["clock_differential"][str(-1 - k)] for k in range(w.s + 1)]
        assert got == [int(x) for x in hist[c - 1]], (model, c, got, hist[c - 1])
        sq, pen = obj[c - 1]
        assert abs(row["sq_loss"] - sq) <= 1e-5 * sq and abs(row["penalised"] - pen) <= 1e-5 * pen, (c, row, sq)
    tot = np.sum(hist, axis=0)
    for k in range(w.s + 1):
        assert rep["clock_differential"][str(-1 - k)] == pytest.approx(tot[k] / tot.sum(), abs=1e-12)


def test_report_essp_freshest_share_closed_form():
    """512 workers, s = 3, 20 clocks: over clocks 5..20 (past the start-up,
    where v >= 0 truncates the delay) the share of reads at differential -1
    is 0.7 within 4 standard deviations of a binomial share."""
    from paper_1410_8043_gb300 import report

    w = workload("tiny").with_(name="tiny_essp_p512", model="essp", P=512, s=3)
    rep = report.run_workload(w)
    fresh = sum(r["clock_differential"]["-1"] for r in rep["per_clock"][4:])
    n = 512 * (w.clocks - 4)
    sd = (0.7 * 0.3 / n) ** 0.5
    assert abs(fresh / n - 0.7) <= 4 * sd, fresh / n
