"""Parity at the full workload sizes, in the launch configuration the
benchmark times (same kernels, grids and data layout).

* mid (480k x 18k, 100M entries, K=100, P=32, SSP s=3) and mid_essp: the
  first clocks compared element by element with the oracle, plus the
  objective over all 100M entries;
* large (10M x 1M, 2B entries, K=64, P=128, SSP s=4): the first clock
  compared element by element (the oracle takes about a minute per clock
  there); set ESSPT_SKIP_LARGE=1 to skip it on a small host.
* the whole 40-clock mid trajectory runs when ESSPT_LONG=1 (several minutes
  of oracle time).
"""
import os

import numpy as np
import pytest

from gen import workload
from oracle import Oracle

pytestmark = pytest.mark.gpu

TOL = 1e-4
_cache = {}


def _data(name):
    if name not in _cache:
        w = workload(name)
        _cache.clear()
        _cache[name] = (w.make_data(), w.partition())
    return _cache[name]


def _parity(name, clocks, obj_every=1):
    from paper_1410_8043_gb300 import esspt

    w = workload(name)
    base = "mid" if name.startswith("mid") else name
    d, part = _data(base)
    t = esspt.Table.for_workload(w, d, part)
    o = Oracle.from_workload(w, d, part)
    worst = []
    for c in range(1, clocks + 1):
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
        o.clock()
        x = o.table()
        g = t.read_table(c).cpu().numpy()
        err = np.abs(g.astype(np.float64) - x) - TOL * (1.0 + np.abs(x))
        worst.append(float(err.max()))
        assert worst[-1] <= 0.0, f"{name} clock {c}: max |err| {np.abs(g - x).max():.3e}"
        del g, x
        if obj_every and c % obj_every == 0:
            gs, gp = t.mf_objective(c, w.lam)
            os_, op = o.objective()
            assert abs(gs - os_) <= 1e-4 * abs(os_) and abs(gp - op) <= 1e-4 * abs(op), (c, gs, os_, gp, op)
    v, clk = t.read_schedule()
    assert clk == clocks + 1
    t.close()
    return worst


def test_mid_ssp_first_clocks():
    _parity("mid", 3)


def test_mid_essp_first_clocks():
    _parity("mid_essp", 2)


@pytest.mark.skipif(os.environ.get("ESSPT_LONG") != "1", reason="set ESSPT_LONG=1 for the 40-clock trajectory")
@pytest.mark.parametrize("name", ["mid", "mid_essp"])
def test_mid_whole_trajectory(name):
    _parity(name, workload(name).clocks, obj_every=5)


@pytest.mark.skipif(os.environ.get("ESSPT_SKIP_LARGE") == "1", reason="ESSPT_SKIP_LARGE=1")
def test_large_first_clock():
    _parity("large", 1, obj_every=0)
