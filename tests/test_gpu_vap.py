"""GPU parity of the VAP read schedule (Sec. 2.1) and of the decaying step
size eta / sqrt(c) of the Sec. 3 theorems, against the fp64 oracle.

VAP compares fp32 max-norms of table differences with its bound, so the
oracle (fp64 norms of fp64 tables) and the GPU take the same decision only
where the norm is not within rounding of the bound: the tests first check,
on the oracle, that every decision they rely on has a relative margin of at
least 1e-3, far above the ~1e-6 gap between the two tables.
"""
import numpy as np
import pytest
import torch

from gen import workload
from oracle import Oracle, OracleConfig

pytestmark = pytest.mark.gpu

TOL = 1e-4
MARGIN = 1e-3


def _esspt():
    from paper_1410_8043_gb300 import esspt

    return esspt


def _viol(g, o):
    return float((np.abs(g - o) - TOL * (1.0 + np.abs(o))).max())


@pytest.mark.parametrize("v0", [0.07, 0.0, 1e30])
def test_vap_tiny_every_clock(v0):
    """Schedule bit-exact and every parameter within tolerance for 20 clocks;
    v0 = 0.07 mixes staleness 0..3, 0 gives BSP and 1e30 the stalest reads."""
    E = _esspt()
    w = workload("tiny").with_(model="vap", s=3, vap_v0=v0)
    d = w.make_data()
    part = w.partition()
    t = E.Table.for_workload(w, d, part)
    o = Oracle.from_workload(w, d, part)
    seen = set()
    for c in range(1, w.clocks + 1):
        v_gpu, clk = t.read_schedule()
        assert clk == c
        o.clock()
        v_or = o.schedule()
        norms, bound = o.vap_norms()
        for k in range(1, min(w.s, c - 1) + 1):
            if 0.0 < bound < 1e20:
                assert abs(norms[k] - bound) > MARGIN * bound, (c, k, norms[k], bound)
        np.testing.assert_array_equal(v_gpu, v_or, err_msg=f"clock {c}")
        seen.add(int(c - 1 - v_or[0]))
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
        g = t.read_table(c).cpu().numpy().astype(np.float64)
        assert _viol(g, o.table()) <= 0.0, f"clock {c}: max |err| {np.abs(g - o.table()).max():.3e}"
    if v0 == 0.07:
        assert seen == {0, 1, 2, 3}
    gs, gp = t.mf_objective(w.clocks, w.lam)
    os_, op = o.objective()
    assert abs(gs - os_) <= 1e-5 * abs(os_) and abs(gp - op) <= 1e-5 * abs(op)
    t.close()


@pytest.mark.parametrize("K,v0", [(48, 0.6), (64, 0.6), (100, 0.8)])
def test_vap_wide_rows_every_clock(K, v0):
    """VAP on the work-list path (K = 48, 64) and on the one-slice-per-lane
    kernel (K = 100), Zipf items, a hot-row cap: schedule bit-exact and every
    parameter within tolerance for 12 clocks, reads of every staleness 0..3."""
    from gen import make_mf_data, minibatch_labels, shard_users

    E = _esspt()
    N, M, n, P, F, s = 500, 60, 20000, 7, 4, 3
    d = make_mf_data(n_users=N, n_items=M, n_obs=n, K=K, seed=3, item_dist="zipf", item_a=1.0, truth_rank=4,
                     truth_var=0.5, noise_var=0.1, init_var=0.05)
    wp, mb = shard_users(N, P, 5), minibatch_labels(n, F, 6)
    eta, lam, cap = 0.01, 0.05, 12
    t = E.Table(N + M, K, P, s, model="vap", vap_v0=v0)
    t.mf_load(d.i, d.j, d.D, mb, wp, N, F)
    t.table_init(np.concatenate([d.L0, d.R0]))
    cfg = OracleConfig(n_users=N, n_items=M, K=K, P=P, s=s, F=F, model="vap", phased=True, seed=8043, eta=eta,
                       lam=lam, cap=cap, vap_v0=v0)
    o = Oracle(cfg, d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    seen = set()
    for c in range(1, 13):
        v_gpu, clk = t.read_schedule()
        assert clk == c
        o.clock()
        v_or = o.schedule()
        norms, bound = o.vap_norms()
        for k in range(1, min(s, c - 1) + 1):
            if 0.0 < bound < 1e20:
                assert abs(norms[k] - bound) > MARGIN * bound, (c, k, norms[k], bound)
        np.testing.assert_array_equal(v_gpu, v_or, err_msg=f"clock {c}")
        seen.add(int(c - 1 - v_or[0]))
        t.mf_sgd_clock(eta, lam, cap)
        g = t.read_table(c).cpu().numpy().astype(np.float64)
        assert _viol(g, o.table()) <= 0.0, f"clock {c}: max |err| {np.abs(g - o.table()).max():.3e}"
    assert seen == {0, 1, 2, 3}
    t.close()


def test_vap_get_inc_clock_by_hand():
    """VAP on the generic GET/INC/CLOCK path with hand-set deltas (s = 2, v0 = 1):
    clock 1 adds 1/2 to row 0, clock 2 adds 1/4 to row 1, clock 3 adds 1/8 to
    row 0, clock 4 adds 2 to row 2.  Bounds 1/sqrt(c):
      c=2: |X1-X0| = 1/2 <= 0.707, v = 0;   c=3: |X2-X0| = 1/2 <= 0.577, v = 0;
      c=4: |X3-X1| = 1/4 <= 1/2, v = 1;     c=5: |X4-X2| = |X4-X3| = 2 > 0.447, v = 4."""
    E = _esspt()
    t = E.Table(8, 4, 2, 2, model="vap", vap_v0=1.0)
    t.table_init(np.zeros((8, 4), np.float32))
    dev = torch.device("cuda")
    incs = [(0, 0.5), (1, 0.25), (0, 0.125), (2, 2.0)]
    want = [0, 0, 0, 1, 4]
    for c in range(1, 6):
        v, clk = t.read_schedule()
        assert clk == c and list(v) == [want[c - 1]] * 2, (c, list(v))
        if c <= len(incs):
            r, x = incs[c - 1]
            t.inc(0, torch.tensor([r], dtype=torch.int32, device=dev), torch.full((1, 4), x, device=dev))
            t.clock()
    t.close()


def test_eta_decay_tiny():
    """eta_c = eta / sqrt(c), passed per clock through the C-ABI, against the
    oracle's decaying step size, 12 clocks of the tiny workload."""
    E = _esspt()
    w = workload("tiny")
    d = w.make_data()
    part = w.partition()
    t = E.Table.for_workload(w, d, part)
    o = Oracle(OracleConfig.from_workload(w, eta_decay=True), d.i, d.j, d.D, part[1], part[0], d.L0, d.R0)
    for c in range(1, 13):
        t.mf_sgd_clock(float(np.float32(w.eta / np.sqrt(c))), w.lam, w.cap)
        o.clock()
        g = t.read_table(c).cpu().numpy().astype(np.float64)
        assert _viol(g, o.table()) <= 0.0, c
    t.close()
