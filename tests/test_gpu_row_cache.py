"""GPU parity of row-granular SSP (Sec. 4 client cache: a clock c_param per
cached row, refreshed only when too stale) against the fp64 oracle: every
parameter after every clock, on the paths of every row width, the chunked
heavy-user path, and the generic GET/INC/CLOCK interface by hand."""
import numpy as np
import pytest
import torch

from gen import make_mf_data, minibatch_labels, shard_users, workload
from oracle import Oracle, OracleConfig

pytestmark = pytest.mark.gpu

TOL = 1e-4


def _esspt():
    from paper_1410_8043_gb300 import esspt

    return esspt


def _run_pair(d, wp, mb, *, P, s, F, eta, lam, cap, clocks, obj_rtol=1e-5):
    E = _esspt()
    N, M, K = d.n_users, d.n_items, d.K
    t = E.Table(N + M, K, P, s, model="ssp_row")
    t.mf_load(d.i, d.j, d.D, mb, wp, N, F)
    t.table_init(np.concatenate([d.L0, d.R0]))
    o = Oracle(OracleConfig(n_users=N, n_items=M, K=K, P=P, s=s, F=F, model="ssp_row", eta=eta, lam=lam, cap=cap),
               d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    for c in range(1, clocks + 1):
        t.mf_sgd_clock(eta, lam, cap)
        o.clock()
        g = t.read_table(c).cpu().numpy().astype(np.float64)
        x = o.table()
        assert float((np.abs(g - x) - TOL * (1 + np.abs(x))).max()) <= 0.0, f"clock {c}: {np.abs(g - x).max():.3e}"
        v, clk = t.read_schedule()
        assert clk == c + 1 and (v == c).all()
    gs, gp = t.mf_objective(clocks, lam)
    os_, op = o.objective()
    assert abs(gs - os_) <= obj_rtol * abs(os_) and abs(gp - op) <= obj_rtol * abs(op)
    t.close()


@pytest.mark.parametrize("s", [1, 3])
def test_row_cache_tiny_every_clock(s):
    """Tiny workload (10 minibatches, so rows are read sporadically), 20 clocks."""
    w = workload("tiny")
    d = w.make_data()
    wp, mb = w.partition()
    _run_pair(d, wp, mb, P=w.P, s=s, F=w.F, eta=w.eta, lam=w.lam, cap=w.cap, clocks=w.clocks)


@pytest.mark.parametrize("K", [16, 48, 100, 132])
def test_row_cache_row_widths(K):
    """The generic, work-list, one-slice-per-lane and wide-row SGD kernels in row mode."""
    d = make_mf_data(n_users=300, n_items=120, n_obs=6000, K=K, seed=K + 1, truth_rank=4, truth_var=0.5,
                     noise_var=0.1, init_var=0.05)
    _run_pair(d, shard_users(300, 5, 1), minibatch_labels(6000, 3, 2), P=5, s=2, F=3, eta=0.02, lam=0.05, cap=0,
              clocks=6)


@pytest.mark.parametrize("K", [32, 64])
def test_row_cache_heavy_users(K):
    """Users with thousands of entries per minibatch take the chunked path."""
    d = make_mf_data(n_users=400, n_items=300, n_obs=40000, K=K, seed=9, user_dist="zipf", user_a=1.5,
                     truth_rank=4, truth_var=0.5, noise_var=0.1, init_var=0.05)
    _run_pair(d, shard_users(400, 3, 8), minibatch_labels(40000, 2, 7), P=3, s=1, F=2, eta=0.002, lam=0.05,
              cap=50, clocks=4)


@pytest.mark.parametrize("K", [64, 100])
def test_row_cache_popular_items(K):
    """Popular items with many replica rows (and, at K = 64, the hot items that
    the work-list kernel sums per warp) while each worker reads its own cached
    version of every row; 6 clocks, sparse minibatches so rows age."""
    n = 200_000
    d = make_mf_data(n_users=2000, n_items=40, n_obs=n, K=K, seed=51, user_dist="zipf", user_a=1.2,
                     item_dist="zipf", item_a=1.5, truth_rank=4, truth_var=0.5, noise_var=0.1, init_var=0.05)
    mb = minibatch_labels(n, 3, 52)
    mx = np.max([np.bincount(d.j[mb == b], minlength=40) for b in range(3)], axis=0)
    assert (-(-mx // 2048)).max() > 8  # at least one item with 16 replica rows
    _run_pair(d, shard_users(2000, 5, 53), mb, P=5, s=2, F=3, eta=0.005, lam=0.05, cap=20, clocks=6)


def test_row_cache_get_by_hand():
    """GET under the row-granular cache, s = 1, rows of 4 values, X0 = 0:
      clock 1: worker 0 reads row 0 (not cached: version 0) and adds 1 to it;
      clock 2: worker 0's copy (version 0 >= c-1-s = 0) still serves: 0;
               worker 1 first reads row 0 at version 1: 1; worker 0 adds 1;
      clock 3: worker 0's copy (0 < 1) is refreshed to version 2: 2;
               worker 1 reads row 0 from its version-1 copy (1) and row 1,
               first read, at version 2 (0): oldest version read 1."""
    E = _esspt()
    dev = torch.device("cuda")
    t = E.Table(6, 4, 2, 1, model="ssp_row")
    t.table_init(np.zeros((6, 4), np.float32))
    ids0 = torch.tensor([0], dtype=torch.int32, device=dev)
    one = torch.ones((1, 4), device=dev)

    def get(p, rows):
        out, ver = t.get(p, torch.tensor(rows, dtype=torch.int32, device=dev), want_version=True)
        return out[:, 0].cpu().numpy().tolist(), ver

    assert get(0, [0]) == ([0.0], 0)
    t.inc(0, ids0, one)
    t.clock()
    assert get(0, [0]) == ([0.0], 0)
    assert get(1, [0]) == ([1.0], 1)
    t.inc(0, ids0, one)
    t.clock()
    assert get(0, [0]) == ([2.0], 2)
    assert get(1, [0, 1]) == ([1.0, 0.0], 1)
    t.close()
