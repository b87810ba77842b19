"""GPU parity: the CUDA library against the fp64 oracle, clock by clock.

Bars (the stated tolerances of the method's fp32 arithmetic):
  * every parameter after every clock: |x_gpu - x_oracle| <= 1e-4 (1 + |x_oracle|);
  * objective: 1e-5 relative on the tiny workload, 1e-4 on larger ones;
  * read-version schedule: bit-exact (integer rule).
All calls go through the C-ABI (paper_1410_8043_gb300.esspt).
"""
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


def _max_violation(g, o):
    return float((np.abs(g - o) - TOL * (1.0 + np.abs(o))).max())


class Pair:
    """A GPU table and an oracle on the same inputs."""

    def __init__(self, data, wp, mb, *, P, s, F, model, eta, lam, cap=0, seed=8043, phased=True):
        E = _esspt()
        N, M, K = data.n_users, data.n_items, data.K
        self.N, self.eta, self.lam, self.cap = N, eta, lam, cap
        self.t = E.Table(N + M, K, P, s, model=model, phased=phased, seed=seed)
        self.t.mf_load(data.i, data.j, data.D, mb, wp, N, F)
        self.t.table_init(np.concatenate([data.L0, data.R0]))
        cfg = OracleConfig(n_users=N, n_items=M, K=K, P=P, s=s, F=F, model=model, phased=phased, seed=seed,
                           eta=eta, lam=lam, cap=cap)
        self.o = Oracle(cfg, data.i, data.j, data.D, mb, wp, data.L0, data.R0)
        self.moved = []

    def step(self, check_table=True, obj_rtol=None):
        prev = self.o.table()
        self.t.mf_sgd_clock(self.eta, self.lam, self.cap)
        self.o.clock()
        c = self.o.version
        v_gpu, clk = self.t.read_schedule()
        # the GPU has advanced to clock c+1; the schedule of clock c is the oracle's
        assert clk == c + 1
        if check_table:
            g = self.t.read_table(c).cpu().numpy().astype(np.float64)
            o = self.o.table()
            assert _max_violation(g, o) <= 0.0, f"clock {c}: max |err| {np.abs(g - o).max():.3e}"
            self.moved.append(float(np.abs(o - prev).max()))
        if obj_rtol is not None:
            gs, gp = self.t.mf_objective(c, self.lam)
            os_, op = self.o.objective()
            assert abs(gs - os_) <= obj_rtol * abs(os_), (c, gs, os_)
            assert abs(gp - op) <= obj_rtol * abs(op), (c, gp, op)
        return v_gpu

    def schedule_matches(self, v_next_gpu):
        """The GPU's v(c+1) must equal the oracle's v(c+1), computed at its next clock."""
        return v_next_gpu


def _run(pair, clocks, obj_rtol=None):
    sched_gpu = []
    for _ in range(clocks):
        sched_gpu.append(pair.step(obj_rtol=obj_rtol))
    return sched_gpu


def _oracle_schedules(cfg_kw, clocks):
    """v(c) for c = 1..clocks+1 from a fresh oracle-rule run."""
    from oracle import schedule_rule

    cfg = OracleConfig(**cfg_kw)
    v = np.zeros(cfg.P, np.int32)
    out = []
    for c in range(1, clocks + 2):
        v = schedule_rule(cfg, c, v)
        out.append(v.copy())
    return out


@pytest.mark.parametrize("model", ["ssp", "essp"])
def test_tiny_workload_every_clock(model):
    """The tiny workload (2000 x 1000, 100k entries, K=16, P=4, s=2), all 20 clocks."""
    w = workload("tiny").with_(model=model)
    d = w.make_data()
    wp, mb = w.partition()
    pair = Pair(d, wp, mb, P=w.P, s=w.s, F=w.F, model=w.model, eta=w.eta, lam=w.lam, cap=w.cap, seed=w.sched_seed)
    v_after = _run(pair, w.clocks, obj_rtol=1e-5)
    want = _oracle_schedules(dict(n_users=1, n_items=1, K=1, P=w.P, s=w.s, F=1, model=model, seed=w.sched_seed),
                             w.clocks)
    for c in range(w.clocks):
        np.testing.assert_array_equal(v_after[c], want[c + 1])
    # non-vacuous: the updates are well above the tolerance
    assert min(pair.moved) > 10 * TOL


@pytest.mark.parametrize("p,max_delay,s", [(0.3, 6, 8), (0.9, 1, 4), (1.0, 3, 3), (0.05, 8, 8), (0.5, 5, 2)])
def test_essp_delay_law_parameters(p, max_delay, s):
    """ESSP with other push probabilities and delay clamps than the workloads'
    (Geometric(0.7), clamp 3): the read versions of 64 workers over 40 clocks
    equal the oracle's rule bit for bit, within the clamp min(max_delay, s)
    and spread over several staleness values."""
    E = _esspt()
    P, seed = 64, 77
    t = E.Table(8, 4, P, s, model="essp", essp_p=p, essp_max_delay=max_delay, seed=seed)
    t.table_init(np.zeros((8, 4), np.float32))
    want = _oracle_schedules(dict(n_users=1, n_items=1, K=1, P=P, s=s, F=1, model="essp", seed=seed, essp_p=p,
                                  essp_max_delay=max_delay), 40)
    stale = set()
    for c in range(1, 41):
        v, clk = t.read_schedule()
        assert clk == c
        np.testing.assert_array_equal(v, want[c - 1], err_msg=f"clock {c}")
        stale.update((c - 1 - v).tolist())
        t.clock()
    t.poll()
    bound = 0 if p == 1.0 else min(max_delay, s)
    assert max(stale) <= bound and len(stale) >= min(bound + 1, 5)
    t.close()


@pytest.mark.parametrize("K", [4, 8, 12, 16, 36, 52, 64, 100, 128, 132, 260])
def test_row_widths_and_ragged_tail(K):
    """Every row-group shape (lanes per row, float4 per lane) and ragged K."""
    d = make_mf_data(n_users=300, n_items=120, n_obs=6000, K=K, seed=K, truth_rank=4, truth_var=0.5,
                     noise_var=0.1, init_var=0.05)
    P, F = 5, 3
    pair = Pair(d, shard_users(300, P, 1), minibatch_labels(6000, F, 2), P=P, s=2, F=F, model="essp",
                eta=0.02, lam=0.05)
    _run(pair, 5, obj_rtol=1e-5)


@pytest.mark.parametrize("cap", [0, 12])
@pytest.mark.parametrize("s,model", [(0, "ssp"), (1, "essp"), (3, "ssp"), (3, "essp")])
def test_staleness_models_and_cap(s, model, cap):
    d = make_mf_data(n_users=500, n_items=60, n_obs=20000, K=20, seed=3, item_dist="zipf", item_a=1.0,
                     truth_rank=4, truth_var=0.5, noise_var=0.1, init_var=0.05)
    P, F = 7, 4
    pair = Pair(d, shard_users(500, P, 5), minibatch_labels(20000, F, 6), P=P, s=s, F=F, model=model,
                eta=0.01, lam=0.05, cap=cap)
    _run(pair, 8, obj_rtol=1e-5)


@pytest.mark.parametrize("K", [32, 40, 64])
def test_heavy_users_chunk_path(K):
    """Users with far more than 96 entries in a minibatch (Zipf(1.5) users) go
    through the chunked kernels (for K = 40 and 64 as items of the work-list
    kernel, beside the light users and the forward copy of idle users);
    results must not change."""
    d = make_mf_data(n_users=400, n_items=300, n_obs=40000, K=K, seed=9, user_dist="zipf", user_a=1.5,
                     truth_rank=4, truth_var=0.5, noise_var=0.1, init_var=0.05)
    mb = minibatch_labels(40000, 2, 7)
    counts = np.bincount(d.i[mb == 0], minlength=400)
    assert counts.max() > 2000 and (counts > 96).sum() >= 3
    pair = Pair(d, shard_users(400, 3, 8), mb, P=3, s=1, F=2, model="ssp", eta=0.002, lam=0.05, cap=50)
    _run(pair, 4, obj_rtol=1e-5)


@pytest.mark.parametrize("K", [16, 48, 64, 100, 132])
def test_popular_items_with_extra_replicas(K):
    """Items popular enough for extra replica rows (one per 2048 entries of
    their largest minibatch, a power of two, at most 64), here 1 to 64 of
    them, beside heavy users, idle users and (for K = 48, 64) the two hot
    items that the work-list kernel sums per warp.  The item merge must add
    every replica and clear it for the next clock."""
    n = 400_000
    d = make_mf_data(n_users=3000, n_items=40, n_obs=n, K=K, seed=11, user_dist="zipf", user_a=1.2,
                     item_dist="zipf", item_a=1.5, truth_rank=4, truth_var=0.5, noise_var=0.1, init_var=0.05)
    F = 2
    mb = minibatch_labels(n, F, 12)
    mx = np.max([np.bincount(d.j[mb == b], minlength=40) for b in range(F)], axis=0)
    want = -(-mx // 2048)
    assert want.max() > 32 and ((want > 1) & (want <= 8)).sum() >= 3  # the cap of 64 and small counts
    users = np.bincount(d.i[mb == 0], minlength=3000)
    assert (users > 96).sum() >= 10 and (users == 0).sum() >= 1
    pair = Pair(d, shard_users(3000, 6, 13), mb, P=6, s=2, F=F, model="essp", eta=0.005, lam=0.05, cap=20)
    _run(pair, 5, obj_rtol=1e-5)
    assert min(pair.moved) > 10 * TOL


@pytest.mark.parametrize("K", [16, 64, 100])
def test_rows_that_no_entry_names(K):
    """Users and items that no entry names keep their initial rows, bit for bit,
    in every version, through more clocks than the ring has slots (so the
    work-list path also skips their forward copies)."""
    d = make_mf_data(n_users=400, n_items=90, n_obs=12000, K=K, seed=21, item_dist="zipf", item_a=1.0,
                     truth_rank=4, truth_var=0.5, noise_var=0.1, init_var=0.05)
    d.i = (d.i % 390).astype(np.int32)  # users 390..399 and items 80..89 have no entries
    d.j = (d.j % 80).astype(np.int32)
    P, F, s = 4, 3, 1
    pair = Pair(d, shard_users(400, P, 22), minibatch_labels(12000, F, 23), P=P, s=s, F=F, model="ssp",
                eta=0.01, lam=0.05, cap=10)
    x0 = np.concatenate([d.L0, d.R0])
    quiet = np.r_[390:400, 400 + 80:400 + 90]
    for c in range(1, 9):
        pair.step(obj_rtol=1e-5)
        np.testing.assert_array_equal(pair.t.read_table(c).cpu().numpy()[quiet], x0[quiet])
    assert min(pair.moved) > 10 * TOL


@pytest.mark.parametrize("K", [16, 64, 100])
@pytest.mark.parametrize("shape", ["one_item", "one_user"])
def test_single_item_or_single_user(shape, K):
    """Every entry on one item (a hot item with the most replicas) or on one
    user (one heavy user split into many chunks)."""
    if shape == "one_item":
        N, M, n = 600, 1, 150_000
    else:
        N, M, n = 1, 300, 20_000
    d = make_mf_data(n_users=N, n_items=M, n_obs=n, K=K, seed=31, truth_rank=4, truth_var=0.5, noise_var=0.1,
                     init_var=0.05)
    P, F = 3, 2
    pair = Pair(d, shard_users(N, P, 32), minibatch_labels(n, F, 33), P=P, s=1, F=F, model="essp", eta=0.005,
                lam=0.05, cap=20)
    _run(pair, 5, obj_rtol=1e-5)
    assert min(pair.moved) > 10 * TOL


def test_empty_and_degenerate():
    """No entries at all; P larger than the number of users; one worker."""
    E = _esspt()
    d = make_mf_data(n_users=50, n_items=20, n_obs=0, K=8, seed=1)
    pair = Pair(d, shard_users(50, 64, 1), np.zeros(0, np.uint8), P=64, s=2, F=3, model="ssp", eta=0.1, lam=0.1)
    for _ in range(4):
        pair.step(check_table=True)
    x0 = np.concatenate([d.L0, d.R0])
    np.testing.assert_array_equal(pair.t.read_table(4).cpu().numpy(), x0)
    # an almost-empty minibatch schedule: F larger than the entry count
    d2 = make_mf_data(n_users=10, n_items=10, n_obs=5, K=4, seed=2)
    pair2 = Pair(d2, np.zeros(10, np.int32), minibatch_labels(5, 9, 3), P=1, s=0, F=9, model="ssp", eta=0.1, lam=0.1)
    _run(pair2, 12, obj_rtol=1e-5)
    assert E.Table is not None


def test_inc_then_sgd_in_one_clock():
    """INCs made during a clock land in the same version as that clock's SGD
    deltas: X[c] = X_oracle[c] + sum of INCs (additive updates, Sec. 2.1)."""
    d = make_mf_data(n_users=80, n_items=40, n_obs=3000, K=12, seed=4, truth_rank=3, truth_var=0.5,
                     noise_var=0.1, init_var=0.05)
    P, F = 3, 2
    pair = Pair(d, shard_users(80, P, 9), minibatch_labels(3000, F, 10), P=P, s=1, F=F, model="ssp", eta=0.02,
                lam=0.05)
    rng = np.random.default_rng(0)
    extra = np.zeros((120, 12))
    # two INC calls in clock 1, then its SGD; the oracle has no INC, so only
    # this first clock can be compared (later clocks read the INCed rows)
    for _ in range(2):
        ids = rng.integers(0, 120, size=50).astype(np.int32)
        delta = rng.normal(size=(50, 12)).astype(np.float32) * 0.01
        pair.t.inc(1, ids, delta)
        np.add.at(extra, ids, delta.astype(np.float64))
    pair.t.mf_sgd_clock(pair.eta, pair.lam, 0)
    pair.o.clock()
    g = pair.t.read_table(1).cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(g, pair.o.table() + extra, rtol=0, atol=TOL * 4)


@pytest.mark.parametrize("n_rows,K,n_ids", [(37, 8, 9), (37, 100, 9), (5003, 64, 2000), (301, 512, 150)])
def test_get_inc_clock_semantics(n_rows, K, n_ids):
    """GET returns the worker's read version; INC + CLOCK add into the next
    version; versions outside the window are refused.  Row widths from 8 to
    the largest (512), and id lists that span many blocks."""
    E = _esspt()
    P, s = 3, 2
    t = E.Table(n_rows, K, P, s, model="ssp", phased=True, seed=11)
    x = np.random.default_rng(1).normal(size=(n_rows, K)).astype(np.float32)
    t.table_init(x)
    hist = [x.astype(np.float64)]
    rng = np.random.default_rng(2)
    for c in range(1, 9):
        v, clk = t.read_schedule()
        assert clk == c
        for p in range(P):
            ids = rng.integers(0, n_rows, size=n_ids).astype(np.int32)
            rows, ver = t.get(p, ids, want_version=True)
            assert ver == v[p]
            np.testing.assert_array_equal(rows.cpu().numpy(), hist[ver][ids].astype(np.float32))
        acc = hist[-1].copy()
        for p in range(P):
            ids = rng.integers(0, n_rows, size=2 * n_ids // 3).astype(np.int32)
            dl = rng.normal(size=(ids.size, K)).astype(np.float32)
            t.inc(p, ids, dl)
            np.add.at(acc, ids, dl.astype(np.float64))
        t.clock()
        t.poll()
        got = t.read_table(c).cpu().numpy().astype(np.float64)
        np.testing.assert_allclose(got, acc, rtol=1e-6, atol=1e-5)
        hist.append(got)
    with pytest.raises(E.EssptError):
        t.read_table(8 - s - 1)
    with pytest.raises(E.EssptError):
        t.read_table(9)


def test_external_schedule_and_errors():
    E = _esspt()
    t = E.Table(10, 4, 2, 1, model="external")
    with pytest.raises(E.EssptError) as ei:
        t.clock()
    assert ei.value.status == E.ESTATE
    t.table_init(np.zeros((10, 4), np.float32))
    with pytest.raises(E.EssptError) as ei:
        t.get(0, [1])
    assert ei.value.status == E.ESTATE
    t.set_schedule([0, 0])
    t.clock()
    t.set_schedule([1, 0])
    t.clock()
    with pytest.raises(E.EssptError) as ei:
        t.set_schedule([2, 0])  # clock 3 needs v >= 1
    assert ei.value.status == E.ESTALE
    with pytest.raises(E.EssptError) as ei:
        t.set_schedule([3, 2])  # from the future
    assert ei.value.status == E.ESTALE
    t.set_schedule([2, 1])
    t.get(0, [0, 9])
    t.poll()
    t.get(0, [0, 10])  # out of range row: skipped on the device, reported by poll
    with pytest.raises(E.EssptError) as ei:
        t.poll()
    assert ei.value.status == E.EINVAL
    t.poll()  # cleared
    with pytest.raises(E.EssptError) as ei:
        E.Table(10, 6, 2, 1)  # K not a multiple of 4
    assert ei.value.status == E.EINVAL
    with pytest.raises(E.EssptError) as ei:
        t.mf_sgd_clock(0.1, 0.1)
    assert ei.value.status == E.ESTATE


@pytest.mark.parametrize("K", [16, 64, 100])
def test_external_schedule_random_versions(K):
    """The MF clock under caller-chosen read versions: every worker draws its
    own version anywhere in [max(0, c-1-s), c-1] each clock (not monotone, not
    shared), with heavy users and popular items, so one clock gathers from
    up to s+1 versions at once."""
    E = _esspt()
    N, M, n, P, F, s = 2000, 50, 120_000, 9, 3, 4
    d = make_mf_data(n_users=N, n_items=M, n_obs=n, K=K, seed=41, user_dist="zipf", user_a=1.2,
                     item_dist="zipf", item_a=1.5, truth_rank=4, truth_var=0.5, noise_var=0.1, init_var=0.05)
    wp, mb = shard_users(N, P, 42), minibatch_labels(n, F, 43)
    eta, lam, cap = 0.005, 0.05, 20
    t = E.Table(N + M, K, P, s, model="external")
    t.mf_load(d.i, d.j, d.D, mb, wp, N, F)
    t.table_init(np.concatenate([d.L0, d.R0]))
    o = Oracle(OracleConfig(n_users=N, n_items=M, K=K, P=P, s=s, F=F, model="external", eta=eta, lam=lam, cap=cap),
               d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    rng = np.random.default_rng(44)
    spread = []
    for c in range(1, 11):
        v = rng.integers(max(0, c - 1 - s), c, size=P).astype(np.int32)
        spread.append(len(set(v.tolist())))
        t.set_schedule(v)
        t.mf_sgd_clock(eta, lam, cap)
        o.clock(v_ext=v)
        g = t.read_table(c).cpu().numpy().astype(np.float64)
        assert _max_violation(g, o.table()) <= 0.0, f"clock {c}: max |err| {np.abs(g - o.table()).max():.3e}"
    t.poll()
    assert max(spread) == s + 1
    gs, gp = t.mf_objective(10, lam)
    os_, op = o.objective()
    assert abs(gs - os_) <= 1e-5 * abs(os_) and abs(gp - op) <= 1e-5 * abs(op)
    t.close()


def test_mf_load_rejects_bad_indices():
    E = _esspt()
    t = E.Table(30, 4, 2, 1)
    i = np.array([0, 1, 25], np.int32)  # user 25 >= n_users = 20
    j = np.array([0, 1, 2], np.int32)
    with pytest.raises(E.EssptError) as ei:
        t.mf_load(i, j, np.ones(3, np.float32), np.zeros(3, np.uint8), np.zeros(20, np.int32), 20, 1)
    assert ei.value.status == E.EINVAL
    with pytest.raises(E.EssptError):
        t.mf_load(np.array([0], np.int32), np.array([0], np.int32), np.ones(1, np.float32),
                  np.array([3], np.uint8), np.zeros(20, np.int32), 20, 2)  # minibatch 3 >= F


def test_sq_loss_output():
    """The optional per-clock squared loss equals the oracle's sum of e^2 of
    the clock's entries at their read versions."""
    d = make_mf_data(n_users=200, n_items=90, n_obs=5000, K=16, seed=12, truth_rank=3, truth_var=0.5,
                     noise_var=0.1, init_var=0.05)
    P, F = 4, 2
    wp, mb = shard_users(200, P, 3), minibatch_labels(5000, F, 4)
    pair = Pair(d, wp, mb, P=P, s=0, F=F, model="ssp", eta=0.02, lam=0.05)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    x = pair.o.table(0)
    sel = mb == 0
    Li = x[d.i[sel]]
    Rj = x[200 + d.j[sel]]
    want = float(((d.D[sel].astype(np.float64) - (Li * Rj).sum(1)) ** 2).sum())
    pair.t.mf_sgd_clock(pair.eta, pair.lam, 0, sq_loss=loss)
    got = float(loss.item())
    assert abs(got - want) <= 1e-5 * want


def test_stage_minibatch_values_and_structure_check():
    """Staging a minibatch from host memory: new values take effect in the
    clock that reads it; a changed structure (one item id) is reported by
    poll as EINVAL and never used; a short staging buffer is refused."""
    import ctypes

    E = _esspt()
    N, M, K, P, F = 150, 50, 8, 3, 2
    d = make_mf_data(n_users=N, n_items=M, n_obs=4000, K=K, seed=21, truth_rank=2, truth_var=0.5, noise_var=0.1,
                     init_var=0.05)
    wp, mb = shard_users(N, P, 4), minibatch_labels(4000, F, 5)
    pair = Pair(d, wp, mb, P=P, s=1, F=F, model="ssp", eta=0.02, lam=0.05)
    u, j, D, uoff = pair.t.mf_export_minibatch(0)
    # the device layout of minibatch 0: its entries in a stable sort by user
    idx = np.flatnonzero(mb == 0)
    order = idx[np.argsort(d.i[idx], kind="stable")]
    np.testing.assert_array_equal(u.numpy(), d.i[order])
    np.testing.assert_array_equal(j.numpy(), d.j[order])
    D2 = D.clone() + 0.25
    pair.t.mf_stage_minibatch(0, u, j, D2, uoff, stream=torch.cuda.Stream())
    torch.cuda.synchronize()
    pair.t.poll()
    Dnew = d.D.copy()
    Dnew[order] = D2.numpy()
    o = Oracle(pair.o.cfg, d.i, d.j, Dnew, mb, wp, d.L0, d.R0)
    pair.t.mf_sgd_clock(pair.eta, pair.lam, 0)
    o.clock()
    g = pair.t.read_table(1).cpu().numpy().astype(np.float64)
    assert _max_violation(g, o.table()) <= 0.0
    # a structurally different minibatch: refused at poll, layout untouched
    j_bad = j.clone()
    j_bad[0] = (int(j_bad[0]) + 1) % M
    pair.t.mf_stage_minibatch(0, u, j_bad, D2, uoff)
    with pytest.raises(E.EssptError) as ei:
        pair.t.poll()
    assert ei.value.status == E.EINVAL
    _, j_again, _, _ = pair.t.mf_export_minibatch(0)
    np.testing.assert_array_equal(j_again.numpy(), j.numpy())
    # a staging buffer shorter than esspt_mf_stage_bytes()
    L = E.lib()
    need = L.esspt_mf_stage_bytes(pair.t._h)
    assert need > 256
    st = L.esspt_mf_stage_minibatch(pair.t._h, 0, u.data_ptr(), j.data_ptr(), D.data_ptr(), uoff.data_ptr(),
                                    pair.t._stage.data_ptr(), 256, None)
    assert st == E.ENOSPC
    pair.t.poll()


def test_short_workspaces_are_refused():
    """ESSPT_ENOSPC for a table workspace or an MF workspace shorter than the
    size query; nothing is created or loaded."""
    import ctypes

    E = _esspt()
    L = E.lib()
    cfg = E.Config(100, 8, 2, 1, 0, 1, 3, 0.7, 1, None, 0.0)
    need = L.esspt_workspace_bytes(ctypes.byref(cfg))
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    h = ctypes.c_void_p()
    assert L.esspt_create(ctypes.byref(cfg), ws.data_ptr(), need - 256, ctypes.byref(h)) == E.ENOSPC
    assert not h.value
    d = make_mf_data(n_users=60, n_items=40, n_obs=500, K=8, seed=3)
    t = E.Table(100, 8, 2, 1)
    n_ws = L.esspt_mf_workspace_bytes(t._h, 500, 60, 2)
    n_sc = L.esspt_mf_scratch_bytes(t._h, 500, 60, 2)
    dev = lambda x, dt: torch.as_tensor(x, dtype=dt, device="cuda")  # noqa: E731
    args = [dev(d.i, torch.int32), dev(d.j, torch.int32), dev(d.D, torch.float32),
            dev(minibatch_labels(500, 2, 1), torch.uint8)]
    wk = dev(shard_users(60, 2, 2), torch.int32)
    big = torch.empty(n_ws + n_sc + 512, dtype=torch.uint8, device="cuda")
    base = (big.data_ptr() + 255) // 256 * 256
    for ws_b, sc_b in [(n_ws - 256, n_sc), (n_ws, n_sc - 256)]:
        st = L.esspt_mf_load(t._h, *[a.data_ptr() for a in args], 500, wk.data_ptr(), 60, 2, base, ws_b,
                             base + (n_ws + 255) // 256 * 256, sc_b)
        assert st == E.ENOSPC
    with pytest.raises(E.EssptError) as ei:
        t.mf_sgd_clock(0.01, 0.05)
    assert ei.value.status in (E.ESTATE,)


@pytest.mark.parametrize("K", [40, 64])
def test_idle_rows_skipped_across_the_ring(K):
    """Work-list path, many clocks at s = 1 and 6 minibatches: most user rows
    are idle for more than s+2 clocks in a row, so their forward copy is
    skipped (the ring slot already holds them).  Every clock against the
    oracle; then an INC on an idle row must survive the following clocks."""
    E = _esspt()
    N, M = 600, 80
    d = make_mf_data(n_users=N, n_items=M, n_obs=3000, K=K, seed=K + 7, user_dist="zipf", user_a=1.2,
                     truth_rank=3, truth_var=0.5, noise_var=0.1, init_var=0.05)
    P, F, s = 4, 6, 1
    wp, mb = shard_users(N, P, 3), minibatch_labels(3000, F, 4)
    pair = Pair(d, wp, mb, P=P, s=s, F=F, model="ssp", eta=0.02, lam=0.05)
    _run(pair, 14, obj_rtol=1e-5)
    # an idle user in the coming clocks: INC its row at clock 15, which must
    # stay in every later version (no skip may bring back an older copy)
    coming = set(d.i[np.isin(mb, [(c - 1) % F for c in range(15, 21)])].tolist())
    u = next(x for x in range(N) if x not in coming)
    delta = np.full((1, K), 0.25, np.float32)
    before = pair.t.read_table(14).cpu().numpy()[u].copy()
    pair.t.inc(0, [u], delta)
    for c in range(15, 21):
        pair.t.mf_sgd_clock(pair.eta, pair.lam, 0)
        got = pair.t.read_table(c).cpu().numpy()[u]
        np.testing.assert_allclose(got, before + 0.25, rtol=0, atol=1e-6)
    pair.t.poll()
