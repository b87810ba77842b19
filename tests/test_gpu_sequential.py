"""GPU parity of the sequential (read-my-writes) clock: each worker walks its
entries in order and sees its own updates of the clock (the per-entry SGD
of Sec. 3.1), against the fp64 oracle's sequential mode, every parameter
after every clock."""
import numpy as np
import pytest

from gen import make_mf_data, minibatch_labels, shard_users, workload
from oracle import Oracle, OracleConfig

pytestmark = pytest.mark.gpu

TOL = 1e-4


def _esspt():
    from paper_1410_8043_gb300 import esspt

    return esspt


def _run(d, wp, mb, *, P, s, F, model, eta, lam, cap, clocks):
    E = _esspt()
    N, M, K = d.n_users, d.n_items, d.K
    t = E.Table(N + M, K, P, s, model=model)
    t.mf_load(d.i, d.j, d.D, mb, wp, N, F)
    t.table_init(np.concatenate([d.L0, d.R0]))
    o = Oracle(OracleConfig(n_users=N, n_items=M, K=K, P=P, s=s, F=F, model=model, eta=eta, lam=lam, cap=cap,
                            sequential=True), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    for c in range(1, clocks + 1):
        v, clk = t.read_schedule()
        t.mf_sgd_clock_sequential(eta, lam, cap)
        o.clock()
        np.testing.assert_array_equal(v, o.schedule())
        g = t.read_table(c).cpu().numpy().astype(np.float64)
        x = o.table()
        assert float((np.abs(g - x) - TOL * (1 + np.abs(x))).max()) <= 0.0, f"clock {c}: {np.abs(g - x).max():.3e}"
    gs, gp = t.mf_objective(clocks, lam)
    os_, op = o.objective()
    assert abs(gs - os_) <= 1e-5 * abs(os_) and abs(gp - op) <= 1e-5 * abs(op)
    t.close()


@pytest.mark.parametrize("model", ["ssp", "essp"])
def test_sequential_tiny(model):
    w = workload("tiny")
    d = w.make_data()
    wp, mb = w.partition()
    _run(d, wp, mb, P=w.P, s=w.s, F=w.F, model=model, eta=w.eta, lam=w.lam, cap=w.cap, clocks=8)


@pytest.mark.parametrize("K", [64, 100, 260])
def test_sequential_row_widths_and_cap(K):
    d = make_mf_data(n_users=200, n_items=80, n_obs=5000, K=K, seed=K + 3, truth_rank=4, truth_var=0.5,
                     noise_var=0.1, init_var=0.05)
    _run(d, shard_users(200, 3, 5), minibatch_labels(5000, 2, 6), P=3, s=1, F=2, model="ssp", eta=0.01,
         lam=0.05, cap=20, clocks=4)


def test_sequential_refused_under_row_cache():
    E = _esspt()
    w = workload("tiny")
    d = w.make_data()
    wp, mb = w.partition()
    t = E.Table(w.n_users + w.n_items, w.K, w.P, w.s, model="ssp_row")
    t.mf_load(d.i, d.j, d.D, mb, wp, w.n_users, w.F)
    t.table_init(np.concatenate([d.L0, d.R0]))
    with pytest.raises(E.EssptError):
        t.mf_sgd_clock_sequential(w.eta, w.lam, w.cap)
    t.close()
