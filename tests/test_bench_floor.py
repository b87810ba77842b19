"""Host logic of bench.py's roofline: the compulsory-bytes model of one clock
against a brute-force count on a small workload, and the kernel-launch count
of each read model."""
import numpy as np

from gen import make_mf_data, minibatch_labels, shard_users


def _brute_floor(w, d, wp, mb, c, v):
    """12 B per entry; 8K bytes per user row (read c-1, write c); 4K bytes per
    stale user row read and per distinct (item, stale version) read."""
    b = (c - 1) % w.F
    idx = np.flatnonzero(mb == b)
    total = 12 * idx.size + 8 * w.K * w.n_users
    users = set()
    items = set()
    for k in idx:
        u, j = int(d.i[k]), int(d.j[k])
        ver = int(v[wp[u]])
        if ver != c - 1:
            users.add(u)
            items.add((j, ver))
    return total + 4 * w.K * (len(users) + len(items)), idx.size


def test_floor_model_matches_brute_force():
    import bench
    from gen.workloads import Workload

    d = make_mf_data(n_users=120, n_items=40, n_obs=3000, K=8, seed=5, truth_rank=2)
    P, F = 4, 3
    wp = shard_users(120, P, 6)
    mb = minibatch_labels(3000, F, 7)
    w = Workload("t", 120, 40, 3000, K=8, P=P, F=F, s=3, model="ssp", clocks=5, eta=0.01, lam=0.05, cap=0)
    m = bench.FloorModel(w, d, wp, mb)
    rng = np.random.default_rng(0)
    for c in range(1, 9):
        v = rng.integers(max(0, c - 1 - w.s), c, size=P).astype(np.int32)
        assert m.bytes(c, v) == _brute_floor(w, d, wp, mb, c, v)


def test_floor_model_work_list_skips_unchanged_idle_rows():
    """On the work-list path (K 36..64) an idle user row unchanged over the last
    s+2 clocks is not merged; every user has a 4-byte change-clock word."""
    import bench
    from gen.workloads import Workload

    N, M, K, P, F, s = 150, 30, 40, 3, 4, 1
    d = make_mf_data(n_users=N, n_items=M, n_obs=400, K=K, seed=8, truth_rank=2)
    wp = shard_users(N, P, 9)
    mb = minibatch_labels(400, F, 10)
    w = Workload("t", N, M, 400, K=K, P=P, F=F, s=s, model="ssp", clocks=12, eta=0.01, lam=0.05, cap=0)
    m = bench.FloorModel(w, d, wp, mb)
    rng = np.random.default_rng(1)
    chg = np.zeros(N, np.int64)
    for c in range(1, 13):
        v = rng.integers(max(0, c - 1 - s), c, size=P).astype(np.int32)
        got = m.bytes(c, v)
        base, n = _brute_floor(w, d, wp, mb, c, v)
        active = np.zeros(N, bool)
        active[d.i[mb == (c - 1) % F]] = True
        skipped = int(np.sum(~active & (c - chg >= s + 2)))
        assert skipped > 0 or c < s + 2
        chg[active] = c
        assert got == (base - 8 * K * skipped + 4 * N, n), c


def test_model_launch_counts():
    import bench
    from gen import workload

    assert bench._model_launches(workload("mid"), 10) == 0
    assert bench._model_launches(workload("mid_essp"), 10) == 0
    assert bench._model_launches(workload("mid_row"), 10) == 1
    # VAP: the norms of clock c+1 take one kernel per 8 candidate versions, plus the schedule.
    w = workload("mid_vap")
    assert bench._model_launches(w, 1) == 2 and bench._model_launches(w, 10) == 2
    assert bench._model_launches(w.with_(s=9), 10) == 3


def test_host_minibatches_are_disjoint_views_of_one_buffer(monkeypatch):
    """bench.py's end-to-end leg exports every minibatch into views of one host
    buffer: each view has the size and dtype the export call checks, and no
    two views overlap."""
    import torch

    import bench
    from gen.workloads import Workload

    class CpuBuffer:
        kind = "test"

        def __init__(self, n_int32):
            self.tensor = torch.zeros(n_int32, dtype=torch.int32)
            self.closed = False

        def close(self):
            self.closed = True

    sizes = {0: 7, 2: 0, 3: 13}
    w = Workload("t", 5, 4, 20, K=8, P=2, F=4, s=1, model="ssp", clocks=3, eta=0.01, lam=0.05, cap=0)

    class FakeTable:
        n_users = w.n_users

        def mf_minibatch_size(self, b):
            return sizes[b]

        def mf_export_minibatch(self, b, out):
            u, j, D, uoff = out
            n = sizes[b]
            assert u.numel() == j.numel() == D.numel() == n and uoff.numel() == w.n_users + 1
            assert u.dtype == j.dtype == uoff.dtype == torch.int32 and D.dtype == torch.float32
            assert all(x.is_contiguous() for x in out)
            u.fill_(100 + b)
            j.fill_(200 + b)
            D.fill_(0.5 + b)
            uoff.copy_(torch.arange(w.n_users + 1, dtype=torch.int32) + b)
            return out

    monkeypatch.setattr(bench, "HostBuffer", CpuBuffer)
    out, buf = bench._export_host_minibatches(FakeTable(), w, sorted(sizes))
    assert buf.tensor.numel() == sum(3 * n + w.n_users + 1 for n in sizes.values())
    spans = []
    base = buf.tensor.data_ptr()
    for b, (u, j, D, uoff) in out.items():
        assert bool((u == 100 + b).all()) and bool((j == 200 + b).all()) and bool((D == 0.5 + b).all())
        assert uoff.tolist() == [x + b for x in range(w.n_users + 1)]
        for x in (u, j, D, uoff):
            if x.numel() == 0:  # an empty view has no address to check
                continue
            lo = x.data_ptr() - base
            spans.append((lo, lo + 4 * x.numel()))
            assert 0 <= lo and lo + 4 * x.numel() <= 4 * buf.tensor.numel()
    spans.sort()
    assert all(a[1] <= b[0] for a, b in zip(spans, spans[1:]))


def test_committed_profiles_match_the_kernel_source():
    """The bench line's roofline.traffic comes from the committed ncu summary
    of each headline kernel, and only while the summary's code digest equals
    that of the kernels' current source: both summaries must be current."""
    import bench

    assert bench._profiled_traffic("sgd_work16_kernel", "large") == 7995646720.0
    assert bench._profiled_traffic("sgd_users32_kernel", "mid") == 692899584.0
    assert bench._profiled_traffic("sgd_users32_kernel", "large") is None


def test_kernel_code_digest_ignores_comments_only():
    """The digest that ties a profile to the kernels' code ignores comments and
    layout, and changes with any token of code."""
    import bench

    base = "int f(int x) {\n  return x + 1;  // one more\n}\n"
    assert bench.kernel_code_digest(base) == bench.kernel_code_digest(
        "/* header */\nint f(int x) {\n    return x + 1;\n}\n")
    assert bench.kernel_code_digest(base) != bench.kernel_code_digest(base.replace("x + 1", "x + 2"))
