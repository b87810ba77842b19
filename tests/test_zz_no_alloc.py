"""The allocation-free per-worker objective, checked through the C-ABI.

esspt_mf_worker_objective_noalloc() serves callers that cannot allocate
device memory: its accumulators are an array built into the library.  Its
per-worker sums must add up to what the existing esspt_mf_objective()
returns, on two calls in a row (the shared array keeps the previous call's
contents, so each call must clear it), and each worker's share must match a
direct fp64 sum over that worker's entries.  Worker counts beyond the
array's 2048 slots are refused.

This file is collected last so that a failure here leaves every other test
already run.
"""
import numpy as np
import pytest

from gen import make_mf_data, minibatch_labels, shard_users, workload

pytestmark = pytest.mark.gpu

RTOL = 1e-5  # the objective tolerance of the other parity tests


def _per_worker_reference(x, d, wp, lam, P, N):
    Li = x[d.i].astype(np.float64)
    Rj = x[N + d.j].astype(np.float64)
    e = d.D.astype(np.float64) - (Li * Rj).sum(1)
    pen = e * e + lam * ((Li * Li).sum(1) + (Rj * Rj).sum(1))
    p = wp[d.i]
    return np.bincount(p, weights=e * e, minlength=P), np.bincount(p, weights=pen, minlength=P)


def test_noalloc_worker_objective_two_calls_in_a_row():
    from paper_1410_8043_gb300 import esspt

    w = workload("tiny")
    d = w.make_data()
    wp, mb = w.partition()
    t = esspt.Table.for_workload(w, d, (wp, mb))
    for _ in range(3):
        t.mf_sgd_clock(w.eta, w.lam, w.cap)
    for version in (3, 2, 3):
        sq, pen = t.mf_worker_objective_noalloc(version, w.lam)
        ref_sq, ref_pen = t.mf_objective(version, w.lam)
        assert sq.shape == (w.P,) and pen.shape == (w.P,)
        assert abs(sq.sum() - ref_sq) <= RTOL * abs(ref_sq)
        assert abs(pen.sum() - ref_pen) <= RTOL * abs(ref_pen)
        x = t.read_table(version).cpu().numpy()
        want_sq, want_pen = _per_worker_reference(x, d, wp, w.lam, w.P, w.n_users)
        np.testing.assert_allclose(sq, want_sq, rtol=RTOL)
        np.testing.assert_allclose(pen, want_pen, rtol=RTOL)
    t.close()


def test_noalloc_refuses_more_workers_than_its_array():
    from paper_1410_8043_gb300 import esspt

    N, M, P = 3000, 50, 2049
    d = make_mf_data(n_users=N, n_items=M, n_obs=4000, K=8, seed=5)
    t = esspt.Table(N + M, 8, P, 1)
    t.mf_load(d.i, d.j, d.D, minibatch_labels(4000, 2, 1), shard_users(N, P, 2), N, 2)
    t.table_init(np.concatenate([d.L0, d.R0]))
    t.mf_sgd_clock(0.01, 0.05, 0)
    with pytest.raises(esspt.EssptError) as ei:
        t.mf_worker_objective_noalloc(1, 0.05)
    assert ei.value.status == esspt.EINVAL and "2048" in str(ei.value)
    t.close()
