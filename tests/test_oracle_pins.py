"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: hand-worked
clocks, closed forms of the schedule, a special case that reduces to plain
gradient descent computed by automatic differentiation, invariants of the
consistency models, and the published SplitMix64 output sequence.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

from gen import ctr_u64 as gen_ctr
from gen import make_mf_data, minibatch_labels, shard_users
from oracle import Oracle, OracleConfig, ctr_u64, schedule_rule

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_cases.json")


def _cases():
    with open(GOLDEN) as f:
        return json.load(f)


def _oracle_from_case(case, cap=None, keep_all=False):
    e = np.array(case["entries"], dtype=np.float64).reshape(-1, 3)
    cfg = OracleConfig(
        n_users=case["n_users"], n_items=case["n_items"], K=case["K"], P=case["P"], s=case["s"],
        F=case["F"], model=case.get("model", "external"), eta=case["eta"], lam=case["lambda"],
        cap=case.get("cap", 0) if cap is None else cap, keep_all=keep_all,
        vap_v0=case.get("vap_v0", 0.0), eta_decay=case.get("eta_decay", False),
        sequential=case.get("sequential", False),
    )
    return Oracle(
        cfg, e[:, 0].astype(np.int32), e[:, 1].astype(np.int32), e[:, 2].astype(np.float32),
        np.array(case.get("minibatch", [0] * e.shape[0]), np.uint8), np.array(case["user_worker"], np.int32),
        np.array(case["L0"], np.float32), np.array(case["R0"], np.float32),
    )


def _frac_table(rows):
    return np.array([[float(Fraction(x)) for x in r] for r in rows], dtype=np.float64)


@pytest.mark.parametrize(
    "name",
    ["single_entry", "stale_k1", "penalty_k2", "hot_row_cap", "vap_single_entry", "eta_decay_single_entry",
     "row_cache_two_workers", "sequential_one_worker"],
)
def test_hand_worked_clocks(name):
    """Sec. 3.1 update rule, stale reads and the Clock() merge, against hand-worked values.

    Cases with the external model give the schedule; the VAP case must choose
    it by its value bound, and the others read version c-1 (s = 0)."""
    case = _cases()[name]
    o = _oracle_from_case(case)
    N = case["n_users"]
    external = case.get("model", "external") == "external"
    for c, v in enumerate(case["schedule"], start=1):
        if external:
            o.clock(v_ext=v)
        else:
            o.clock()
            assert list(o.schedule()) == v, (c, list(o.schedule()), v)
        want = case["versions"].get(str(c))
        if want is None:
            continue
        for p, r, ver in case.get("row_versions", {}).get(str(c), []):
            assert o.row_version(p, r) == ver, (c, p, r)
        x = o.table()
        np.testing.assert_allclose(x[:N], _frac_table(want["L"]), rtol=0, atol=case["tol"])
        np.testing.assert_allclose(x[N:], _frac_table(want["R"]), rtol=0, atol=case["tol"])
    for ver, (sq, pen) in case.get("objective", {}).items():
        got = o.objective(int(ver))
        assert got[0] == float(Fraction(sq)) and got[1] == float(Fraction(pen))


@pytest.mark.parametrize("name", ["single_entry", "stale_k1", "penalty_k2", "sequential_one_worker"])
def test_hand_worked_clock_losses(name):
    """The clock's own squared loss (sum of e^2 over its entries, each at its
    read version) against the hand-derived residuals of each clock."""
    case = _cases()[name]
    o = _oracle_from_case(case)
    external = case.get("model", "external") == "external"
    want = case["clock_loss"]
    for c, v in enumerate(case["schedule"], start=1):
        o.clock(v_ext=v) if external else o.clock()
        if str(c) in want:
            assert o.clock_loss() == float(Fraction(want[str(c)])), (name, c)


def test_clock_loss_full_batch_bsp_is_squared_loss():
    """With one minibatch (F = 1) and s = 0 every entry is read at X[c-1], so
    the clock's loss is the squared loss J of version c-1 (Sec. 5)."""
    d = make_mf_data(n_users=40, n_items=25, n_obs=600, K=6, seed=13, truth_rank=2)
    P = 3
    cfg = OracleConfig(n_users=40, n_items=25, K=6, P=P, s=0, F=1, model="essp", eta=0.01, lam=0.05)
    o = Oracle(cfg, d.i, d.j, d.D, np.zeros(600, np.uint8), shard_users(40, P, 2), d.L0, d.R0)
    for c in range(1, 5):
        want = o.objective(c - 1)[0]
        o.clock()
        assert o.clock_loss() == pytest.approx(want, rel=1e-12), c


def test_bound_violation_rejected():
    """A read that misses updates of clocks <= c-s-1 breaks the SSP condition (Sec. 2.2)."""
    case = _cases()["stale_k1"]
    o = _oracle_from_case(case)
    o.clock(v_ext=case["schedule"][0])
    o.clock(v_ext=case["schedule"][1])
    before = o.table()
    with pytest.raises(ValueError):
        o.clock(v_ext=case["bad_schedule_clock3"])
    assert o.version == 2
    np.testing.assert_array_equal(o.table(), before)
    with pytest.raises(ValueError):
        o.clock(v_ext=[3, 2])  # a version from the future


def test_splitmix64_published_sequence():
    """SplitMix64 from state 0 starts 0xe220a8397b1dcdaf, 0x6e789e6aa1b965f4,
    0x06c45d188009454f (Steele, Lea and Flood 2014 reference generator)."""
    want = [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    assert [ctr_u64(0, 0, k) for k in range(3)] == want
    assert [int(gen_ctr(0, 0, k)) for k in range(3)] == want
    idx = np.arange(0, 5000, 37, dtype=np.uint64)
    for seed, stream in [(8043, 101), (1, 102), (2**64 - 1, 7)]:
        g = gen_ctr(seed, stream, idx)
        assert [int(x) for x in g] == [ctr_u64(seed, stream, int(k)) for k in idx]


def _run_schedule(cfg, clocks):
    v = np.zeros(cfg.P, np.int32)
    out = []
    for c in range(1, clocks + 1):
        v = schedule_rule(cfg, c, v)
        assert v is not None
        out.append(v.copy())
    return np.array(out)


@pytest.mark.parametrize("model", ["ssp", "essp"])
@pytest.mark.parametrize("s", [0, 1, 2, 3, 8])
@pytest.mark.parametrize("phased", [True, False])
def test_schedule_bound_monotone_window(model, s, phased):
    """Formal SSP bound (Sec. 3): a read at clock c sees every update of clocks
    1..c-s-1 and none from the future; reads never go backwards; at most s
    clocks of P workers' updates are missing, inside the P(2s+1) window of Lemma 4."""
    P = 37
    cfg = OracleConfig(n_users=1, n_items=1, K=1, P=P, s=s, F=1, model=model, phased=phased, seed=99)
    sched = _run_schedule(cfg, 60)
    c = np.arange(1, 61)[:, None]
    assert (sched <= c - 1).all()
    assert (sched >= np.maximum(0, c - 1 - s)).all()
    assert (np.diff(sched, axis=0) >= 0).all()
    missing = (c - 1 - sched) * P
    assert (missing <= P * (2 * s + 1)).all()


@pytest.mark.parametrize("model", ["ssp", "essp"])
def test_bsp_special_case(model):
    """s = 0 is BSP: every read is the previous clock, clock differential -1 (Fig. 1)."""
    cfg = OracleConfig(n_users=1, n_items=1, K=1, P=64, s=0, F=1, model=model, seed=5)
    sched = _run_schedule(cfg, 30)
    c = np.arange(1, 31)[:, None]
    assert ((sched - c) == -1).all()


@pytest.mark.parametrize("s", [1, 3, 5])
def test_ssp_lazy_staleness_exactly_uniform(s):
    """SSP lazy pull refreshes only when forced (Sec. 2.2), so once c > s each
    worker's staleness cycles through 0..s: exactly uniform on {0..s}."""
    P = 16
    cfg = OracleConfig(n_users=1, n_items=1, K=1, P=P, s=s, F=1, model="ssp", seed=17)
    C = 1 + s + 20 * (s + 1)
    sched = _run_schedule(cfg, C)
    c = np.arange(1, C + 1)[:, None]
    st = (c - 1 - sched)[s + 1:]
    for p in range(P):
        counts = np.bincount(st[:, p], minlength=s + 1)
        assert (counts == 20).all()
    # a refresh jumps to the newest version
    jumps = np.diff(sched, axis=0) > 0
    assert ((sched[1:] == (c[1:] - 1)) | ~jumps).all()


def test_essp_stationary_staleness_closed_form():
    """ESSP (Sec. 2.2, Sec. 4): with delays d ~ Geometric(0.7) clamped to 3 and
    monotone reads, staleness obeys st_c = min(d_c, st_{c-1} + 1), whose
    stationary law is P(st >= k) = 0.3^(k(k+1)/2): (0.7, 0.273, 0.026271, 0.000729)."""
    P = 1024
    cfg = OracleConfig(n_users=1, n_items=1, K=1, P=P, s=3, F=1, model="essp", seed=8043)
    C = 1200
    sched = _run_schedule(cfg, C)
    c = np.arange(1, C + 1)[:, None]
    st = (c - 1 - sched)[20:].ravel()
    n = st.size
    want = np.array([0.7, 0.273, 0.026271, 0.000729])
    got = np.bincount(st, minlength=4)[:4]
    assert got.sum() == n
    sigma = np.sqrt(n * want * (1 - want))
    assert (np.abs(got - n * want) < 5 * sigma).all(), (got / n, want)
    assert abs(st.mean() - 0.327729) < 5 * st.std() / np.sqrt(n) * 3


@pytest.mark.parametrize("p", [0.5, 0.3])
def test_essp_stationary_staleness_other_laws(p):
    """The same closed form for other push probabilities, with the clamp at 8
    out of the way: P(st >= k) = (1-p)^(k(k+1)/2), since st_c >= k needs
    d_c >= k and st_{c-1} >= k-1."""
    P, C, q = 1024, 1200, 1.0 - p
    cfg = OracleConfig(n_users=1, n_items=1, K=1, P=P, s=8, F=1, model="essp", seed=8043, essp_p=p,
                       essp_max_delay=8)
    sched = _run_schedule(cfg, C)
    c = np.arange(1, C + 1)[:, None]
    st = (c - 1 - sched)[30:].ravel()
    n = st.size
    ge = np.array([q ** (k * (k + 1) / 2) for k in range(7)])
    want = ge[:6] - ge[1:7]  # P(st = k), k = 0..5
    got = np.bincount(st, minlength=9)[:6]
    sigma = np.sqrt(n * want * (1 - want))
    assert (np.abs(got - n * want) < 5 * sigma).all(), (got / n, want)


def test_essp_delay_thresholds_exact():
    """The ESSP delay rule's 32-bit thresholds are floor(0.3^k 2^32) for the
    Geometric(0.7) delay (failures before the first success), computed here
    in exact rational arithmetic."""
    from oracle import essp_thresholds

    cfg = OracleConfig(n_users=1, n_items=1, K=1, P=1, s=3, F=1, model="essp", essp_p=0.7, essp_max_delay=3)
    want = [int(Fraction(3, 10) ** k * 2 ** 32) for k in (1, 2, 3)]
    assert want == [1288490188, 386547056, 115964116]
    assert essp_thresholds(cfg) == want


@pytest.mark.parametrize("p", ["0.5", "0.3", "0.05", "0.9", "1"])
def test_essp_delay_thresholds_other_laws(p):
    """The same thresholds for other push probabilities and a clamp of 8:
    floor((1-p)^k 2^32) from the decimal p in exact rational arithmetic
    (p = 1 gives no delay: every threshold 0; p = 0.5 gives 2^(32-k))."""
    from oracle import essp_thresholds

    cfg = OracleConfig(n_users=1, n_items=1, K=1, P=1, s=8, F=1, model="essp", essp_p=float(p), essp_max_delay=8)
    q = 1 - Fraction(p)
    want = [int(q ** k * 2 ** 32) for k in range(1, 9)]
    assert essp_thresholds(cfg) == want
    if p == "0.5":
        assert want == [2 ** (32 - k) for k in range(1, 9)]
    if p == "1":
        assert want == [0] * 8


def test_essp_clamped_by_s():
    """For s < 3 the delay is clamped to s, so ESSP never leaves the SSP window."""
    for s in (1, 2):
        cfg = OracleConfig(n_users=1, n_items=1, K=1, P=256, s=s, F=1, model="essp", seed=3)
        sched = _run_schedule(cfg, 400)
        c = np.arange(1, 401)[:, None]
        st = (c - 1 - sched)[10:]
        assert st.max() == s and st.min() == 0


def _small_data(n_users=40, n_items=25, n_obs=600, K=4, seed=7, noise_var=0.1):
    return make_mf_data(n_users=n_users, n_items=n_items, n_obs=n_obs, K=K, seed=seed,
                        truth_rank=3, truth_var=0.5, noise_var=noise_var, init_var=0.1)


def _autograd_gd_clock(x, d, rows_mask, eta, lam, N):
    """One step x <- x - eta * grad of 1/2 sum_k [(D_k - L_i.R_j)^2 + lam(|L_i|^2+|R_j|^2)]
    over the entries selected by rows_mask, by torch autograd in fp64."""
    import torch

    X = torch.tensor(x, dtype=torch.float64, requires_grad=True)
    i = torch.tensor(d.i[rows_mask].astype(np.int64))
    j = torch.tensor(d.j[rows_mask].astype(np.int64)) + N
    D = torch.tensor(d.D[rows_mask].astype(np.float64))
    Li, Rj = X[i], X[j]
    f = 0.5 * (((D - (Li * Rj).sum(1)) ** 2).sum() + lam * ((Li ** 2).sum() + (Rj ** 2).sum()))
    (g,) = torch.autograd.grad(f, X)
    return g.numpy()


def test_s0_p1_is_minibatch_gradient_descent():
    """With s = 0 and one worker, a clock is one step of minibatch gradient
    descent on the l2-penalised squared loss of that minibatch (Sec. 3.1)."""
    d = _small_data()
    F = 3
    mb = minibatch_labels(d.n_obs, F, 11)
    eta, lam = 0.02, 0.05
    cfg = OracleConfig(n_users=d.n_users, n_items=d.n_items, K=d.K, P=1, s=0, F=F, eta=eta, lam=lam)
    o = Oracle(cfg, d.i, d.j, d.D, mb, np.zeros(d.n_users, np.int32), d.L0, d.R0)
    x = np.concatenate([d.L0, d.R0]).astype(np.float64)
    for c in range(1, 8):
        g = _autograd_gd_clock(x, d, mb == (c - 1) % F, eta, lam, d.n_users)
        x = x - eta * g
        o.clock()
        np.testing.assert_allclose(o.table(), x, rtol=1e-12, atol=1e-13)


def test_stale_reads_are_gradients_at_read_version():
    """Under any schedule within the bound, clock c adds, for each worker p,
    -eta * grad of p's minibatch loss evaluated at X[v_p(c)] (Sec. 3 SSP:
    u_{p,c} = G(x~_{p,c}); no read-my-writes)."""
    d = _small_data()
    P, s, F = 3, 2, 2
    wp = shard_users(d.n_users, P, 21)
    mb = minibatch_labels(d.n_obs, F, 22)
    eta, lam = 0.03, 0.1
    cfg = OracleConfig(n_users=d.n_users, n_items=d.n_items, K=d.K, P=P, s=s, F=F, model="essp",
                       seed=4, eta=eta, lam=lam, keep_all=True)
    o = Oracle(cfg, d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    hist = [o.table(0)]
    for c in range(1, 10):
        o.clock()
        v = o.schedule()
        want = hist[c - 1].copy()
        for p in range(P):
            sel = (mb == (c - 1) % F) & (wp[d.i] == p)
            want -= eta * _autograd_gd_clock(hist[v[p]], d, sel, eta, lam, d.n_users)
        np.testing.assert_allclose(o.table(), want, rtol=1e-12, atol=1e-13)
        hist.append(o.table())


def test_s0_invariant_to_workers_and_model():
    """At s = 0 every worker reads the previous clock, so the trajectory does not
    depend on P or on the consistency model (BSP, Fig. 1)."""
    d = _small_data()
    mb = minibatch_labels(d.n_obs, 4, 5)
    ref = None
    for P in (1, 3, 8):
        for model in ("ssp", "essp"):
            cfg = OracleConfig(n_users=d.n_users, n_items=d.n_items, K=d.K, P=P, s=0, F=4, model=model)
            o = Oracle(cfg, d.i, d.j, d.D, mb, shard_users(d.n_users, P, 1), d.L0, d.R0)
            for _ in range(6):
                o.clock()
            if ref is None:
                ref = o.table()
            else:
                np.testing.assert_array_equal(o.table(), ref)


@pytest.mark.parametrize(
    "model,extra",
    [("ssp", {}), ("essp", {}), ("vap", {"vap_v0": 0.3}), ("ssp_row", {}), ("ssp", {"sequential": True}),
     ("essp", {"sequential": True})],
)
def test_ring_equals_unbounded_history(model, extra):
    """An (s+2)-slot version ring gives the same tables as keeping every
    version: no read model ever needs a version outside the ring."""
    d = _small_data()
    P, s, F = 5, 3, 3
    wp, mb = shard_users(d.n_users, P, 2), minibatch_labels(d.n_obs, F, 3)
    kw = dict(n_users=d.n_users, n_items=d.n_items, K=d.K, P=P, s=s, F=F, model=model, eta=0.02, **extra)
    a = Oracle(OracleConfig(**kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    b = Oracle(OracleConfig(keep_all=True, **kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    for _ in range(25):
        a.clock()
        b.clock()
        np.testing.assert_array_equal(a.schedule(), b.schedule())
        np.testing.assert_array_equal(a.table(), b.table())
    for ver in range(25 - s - 1, 26):
        np.testing.assert_array_equal(a.table(ver), b.table(ver))
    with pytest.raises(ValueError):
        a.table(25 - s - 2)


@pytest.mark.parametrize("s,P", [(0, 1), (0, 4), (2, 1), (2, 4)])
def test_objective_nonincreasing_noise_free(s, P):
    """Full-batch (F = 1), small step, noise-free data: the penalised objective
    decreases every clock (descent lemma), with or without staleness."""
    d = _small_data(noise_var=0.0)
    cfg = OracleConfig(n_users=d.n_users, n_items=d.n_items, K=d.K, P=P, s=s, F=1, model="ssp",
                       eta=0.002, lam=0.01)
    o = Oracle(cfg, d.i, d.j, d.D, np.zeros(d.n_obs, np.uint8), shard_users(d.n_users, P, 8), d.L0, d.R0)
    prev = o.objective()[1]
    for _ in range(40):
        o.clock()
        cur = o.objective()[1]
        assert cur <= prev
        prev = cur


def test_objective_zero_on_exact_fit():
    """J = 0 when L_i.R_j reproduces every entry; then J_lambda is lambda times
    the squared norms of the touched rows, counted once per entry."""
    rng = np.random.default_rng(0)
    N, M, K = 6, 5, 3
    L = rng.integers(-2, 3, size=(N, K)).astype(np.float32)
    R = rng.integers(-2, 3, size=(M, K)).astype(np.float32)
    i = np.array([0, 1, 2, 3, 4, 5, 0, 2], np.int32)
    j = np.array([0, 1, 2, 3, 4, 0, 4, 4], np.int32)
    D = np.array([np.dot(L[a], R[b]) for a, b in zip(i, j)], np.float32)
    cfg = OracleConfig(n_users=N, n_items=M, K=K, P=1, s=0, F=1, lam=0.25)
    o = Oracle(cfg, i, j, D, np.zeros(8, np.uint8), np.zeros(N, np.int32), L, R)
    sq, pen = o.objective()
    assert sq == 0.0
    norms = sum(float((L[a] ** 2).sum() + (R[b] ** 2).sum()) for a, b in zip(i, j))
    assert pen == 0.25 * norms


def test_cap_scales_only_hot_rows():
    """The hot-row step cap scales row r's summed clock delta by min(1, C/n_r),
    with n_r counted independently here; other rows are untouched."""
    d = _small_data(n_users=30, n_items=6, n_obs=500)
    mb = minibatch_labels(d.n_obs, 2, 9)
    kw = dict(n_users=d.n_users, n_items=d.n_items, K=d.K, P=2, s=1, F=2, eta=0.01)
    wp = shard_users(d.n_users, 2, 4)
    a = Oracle(OracleConfig(cap=0, **kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    b = Oracle(OracleConfig(cap=20, **kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    x0 = a.table()
    a.clock()
    b.clock()
    sel = mb == 0
    n = np.concatenate([np.bincount(d.i[sel], minlength=d.n_users),
                        np.bincount(d.j[sel], minlength=d.n_items)])
    scale = np.minimum(1.0, 20.0 / np.maximum(n, 1))
    assert (n > 20).sum() >= 3  # the cap binds on item rows
    np.testing.assert_allclose(b.table() - x0, scale[:, None] * (a.table() - x0), rtol=1e-12, atol=1e-15)


def _vap_pair(v0, s=3, clocks=8):
    """A VAP oracle and an external-schedule oracle on the same small problem."""
    d = make_mf_data(n_users=300, n_items=200, n_obs=6000, K=8, seed=77, truth_rank=4, truth_var=0.25, noise_var=0.1)
    wp = shard_users(300, 4, 78)
    mb = minibatch_labels(6000, 3, 79)
    kw = dict(n_users=300, n_items=200, K=8, P=4, s=s, F=3, eta=0.02, lam=0.05)
    vap = Oracle(OracleConfig(model="vap", vap_v0=v0, **kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    ext = Oracle(OracleConfig(model="external", **kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    return vap, ext, s, clocks


@pytest.mark.parametrize("v0,stalest", [(0.0, False), (1e300, True)])
def test_vap_limits_reduce_to_fixed_schedules(v0, stalest):
    """VAP (Sec. 2.1) at its two limits: a zero value bound admits no update in
    transit, which is BSP (v = c-1, the s = 0 read of Sec. 2.2); an unbounded
    one admits every version in the window, so each clock reads the stalest,
    max(0, c-1-s).  Both runs must match the external-schedule oracle bit for bit."""
    vap, ext, s, clocks = _vap_pair(v0)
    for c in range(1, clocks + 1):
        want = max(0, c - 1 - s) if stalest else c - 1
        vap.clock()
        ext.clock(v_ext=np.full(4, want, np.int32))
        assert list(vap.schedule()) == [want] * 4, c
        np.testing.assert_array_equal(vap.table(), ext.table())
    norms, bound = vap.vap_norms()
    assert bound == v0 / np.sqrt(clocks)
    assert norms[0] == 0.0 and (norms[1:] > 0).all()


def test_row_cache_at_s0_is_bsp():
    """Row-granular SSP (Sec. 4 client cache) with s = 0 must refresh every row
    it reads to version c-1 each clock: the BSP schedule, bit for bit."""
    d = make_mf_data(n_users=300, n_items=200, n_obs=6000, K=8, seed=77, truth_rank=4, truth_var=0.25, noise_var=0.1)
    wp = shard_users(300, 4, 78)
    mb = minibatch_labels(6000, 3, 79)
    kw = dict(n_users=300, n_items=200, K=8, P=4, s=0, F=3, eta=0.02, lam=0.05)
    row = Oracle(OracleConfig(model="ssp_row", **kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    ext = Oracle(OracleConfig(model="external", **kw), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    for c in range(1, 7):
        row.clock()
        ext.clock(v_ext=np.full(4, c - 1, np.int32))
        np.testing.assert_array_equal(row.table(), ext.table())


def _small_seq_problem(n_users, n_items, n_obs, P, F, seed):
    d = make_mf_data(n_users=n_users, n_items=n_items, n_obs=n_obs, K=8, seed=seed, truth_rank=4, truth_var=0.25,
                     noise_var=0.1)
    return d, shard_users(n_users, P, seed + 1), minibatch_labels(n_obs, F, seed + 2)


def test_sequential_is_textbook_sgd_for_one_worker():
    """With one worker, s = 0 and one minibatch, the sequential clock is plain
    sequential SGD (Sec. 3.1 applied entry by entry, in place): users in
    ascending id, a user's entries in input order."""
    d, _, _ = _small_seq_problem(40, 30, 400, 1, 1, 31)
    wp = np.zeros(40, np.int32)
    mb = np.zeros(400, np.uint8)
    eta, lam = 0.03, 0.05
    o = Oracle(OracleConfig(n_users=40, n_items=30, K=8, P=1, s=0, F=1, model="ssp", eta=eta, lam=lam,
                            sequential=True), d.i, d.j, d.D, mb, wp, d.L0, d.R0)
    L = d.L0.astype(np.float64).copy()
    R = d.R0.astype(np.float64).copy()
    order = sorted(range(400), key=lambda k: (int(d.i[k]), k))
    for c in range(1, 4):
        o.clock()
        for k in order:
            u, j = int(d.i[k]), int(d.j[k])
            e = float(d.D[k]) - float(L[u] @ R[j])
            gl = eta * (e * R[j] - lam * L[u])
            gr = eta * (e * L[u] - lam * R[j])
            L[u] += gl
            R[j] += gr
        x = o.table()
        np.testing.assert_allclose(x[:40], L, rtol=0, atol=1e-12)
        np.testing.assert_allclose(x[40:], R, rtol=0, atol=1e-12)


def test_sequential_equals_minibatch_with_one_entry_per_worker():
    """If no worker has two entries in a clock, reading one's own writes
    changes nothing: the sequential and minibatch clocks agree (to the order
    of the fp64 sums)."""
    n = 60
    d, _, _ = _small_seq_problem(n, 20, n, n, 1, 41)
    i = np.arange(n, dtype=np.int32)  # one entry per user, each user its own worker
    wp = np.arange(n, dtype=np.int32)
    mb = np.zeros(n, np.uint8)
    kw = dict(n_users=n, n_items=20, K=8, P=n, s=2, F=1, model="ssp", phased=True, eta=0.05, lam=0.05)
    seq = Oracle(OracleConfig(sequential=True, **kw), i, d.j, d.D, mb, wp, d.L0, d.R0)
    bat = Oracle(OracleConfig(**kw), i, d.j, d.D, mb, wp, d.L0, d.R0)
    for _ in range(5):
        seq.clock()
        bat.clock()
        np.testing.assert_array_equal(seq.schedule(), bat.schedule())
        np.testing.assert_allclose(seq.table(), bat.table(), rtol=1e-13, atol=1e-15)
