"""The MF-SGD workloads: data recipe plus the consistency-model parameters.

* tiny:  2,000 x 1,000, 100k uniform entries, truth rank 16, rank-16 model,
         4 workers, 1/10 of each shard per clock, SSP s=2, 20 clocks.
* mid:   480k x 18k, 100M entries (Netflix-shaped, Sec. 5), Zipf(1.0) items,
         uniform users, integer ratings 1..5, rank-100 model, 32 workers,
         1/20 per clock, SSP s=3, 40 clocks.
* mid_essp: the mid data under ESSP (eager push), Geometric(0.7) delays
         clamped to [0, 3].
* mid_vap: the mid data under the VAP value bound 0.3 / sqrt(c), s=3.
* mid_row: the mid data under row-granular SSP (per-row cached versions), s=3.
* large: 10M x 1M, 2B entries, Zipf(1.1) users and items, rank-64 model,
         128 workers, 1/50 per clock, SSP s=4, 20 clocks.
* large_s: large's distributions at a fifth of its rows and per-clock entries
         (2M x 200k, 80M entries, 1/10 per clock): the small profiling case.
* sweep: the mid data with s in {0,1,2,4,8} x P in {1,8,64,512} x {SSP, ESSP},
         20 clocks each.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

from .synth import MFData, make_mf_data, minibatch_labels, shard_users

DATA_SEED = 1410
SCHED_SEED = 8043


@dataclass(frozen=True)
class Workload:
    name: str
    n_users: int
    n_items: int
    n_obs: int
    K: int
    P: int
    F: int
    s: int
    model: str  # "ssp" (lazy pull), "essp" (eager push), "vap" (value bound), "ssp_row" (row cache)
    clocks: int
    eta: float
    lam: float
    # Hot-row step cap C (0 = off): a row with n > C entries in a clock has
    # its summed update scaled by C/n.  Summed minibatch updates at the
    # workloads' step size are unstable on Zipf-popular items without it; C =
    # 20 keeps eta*C*|L|^2 well inside the stability range of gradient
    # descent with s clocks of delay (about 2 sin(pi / (2(2s+1)))).
    cap: int
    data: dict = field(default_factory=dict)
    data_seed: int = DATA_SEED
    sched_seed: int = SCHED_SEED
    essp_p: float = 0.7
    essp_max_delay: int = 3
    vap_v0: float = 0.0  # "vap": initial value bound v0 (bound v0 / sqrt(c) at clock c)

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    def make_data(self, n_obs: int | None = None) -> MFData:
        return make_mf_data(
            n_users=self.n_users,
            n_items=self.n_items,
            n_obs=self.n_obs if n_obs is None else n_obs,
            K=self.K,
            seed=self.data_seed,
            **self.data,
        )

    def workers(self):
        """user -> worker, int32[N]."""
        return shard_users(self.n_users, self.P, self.data_seed + 1)

    def minibatches(self):
        """entry -> minibatch, uint8[n_obs]."""
        return minibatch_labels(self.n_obs, self.F, self.data_seed + 2)

    def partition(self):
        """(user -> worker int32[N], entry -> minibatch uint8[n_obs])."""
        return self.workers(), self.minibatches()

    @property
    def ratings_per_clock(self) -> float:
        return self.n_obs / self.F


_MID_DATA = dict(
    item_dist="zipf",
    item_a=1.0,
    truth_rank=32,
    truth_var=32 ** -0.5,
    noise_var=0.8,
    offset=3.6,
    integer_1_5=True,
)

WORKLOADS = {
    "tiny": Workload(
        "tiny", 2000, 1000, 100_000, K=16, P=4, F=10, s=2, model="ssp", clocks=20,
        eta=0.01, lam=0.05, cap=0,
        data=dict(truth_rank=16, truth_var=0.25, noise_var=0.1),
    ),
    "mid": Workload(
        "mid", 480_000, 18_000, 100_000_000, K=100, P=32, F=20, s=3, model="ssp",
        clocks=40, eta=0.005, lam=0.05, cap=20, data=_MID_DATA,
    ),
    "mid_essp": Workload(
        "mid_essp", 480_000, 18_000, 100_000_000, K=100, P=32, F=20, s=3, model="essp",
        clocks=40, eta=0.005, lam=0.05, cap=20, data=_MID_DATA,
    ),
    # VAP read schedule (Sec. 2.1) on the mid data: v0 = 0.3 gives reads of
    # staleness 0..3 over the first clocks, then a mix of 2 and 3.
    "mid_vap": Workload(
        "mid_vap", 480_000, 18_000, 100_000_000, K=100, P=32, F=20, s=3, model="vap",
        clocks=40, eta=0.005, lam=0.05, cap=20, data=_MID_DATA, vap_v0=0.3,
    ),
    # Row-granular SSP (Sec. 4 client cache, a c_param per row) on the mid data.
    "mid_row": Workload(
        "mid_row", 480_000, 18_000, 100_000_000, K=100, P=32, F=20, s=3, model="ssp_row",
        clocks=40, eta=0.005, lam=0.05, cap=20, data=_MID_DATA,
    ),
    "large": Workload(
        "large", 10_000_000, 1_000_000, 2_000_000_000, K=64, P=128, F=50, s=4,
        model="ssp", clocks=20, eta=0.005, lam=0.05, cap=20,
        data=dict(user_dist="zipf", user_a=1.1, item_dist="zipf", item_a=1.1,
                  truth_rank=32, truth_var=32 ** -0.5, noise_var=0.5),
    ),
    # The large workload's distributions at a fifth of its rows and entries
    # per clock (2M x 200k, 8M entries per clock): the small case for ncu
    # counter captures of the K=64 kernels, a few GB on the device.
    "large_s": Workload(
        "large_s", 2_000_000, 200_000, 80_000_000, K=64, P=128, F=10, s=4,
        model="ssp", clocks=20, eta=0.005, lam=0.05, cap=20,
        data=dict(user_dist="zipf", user_a=1.1, item_dist="zipf", item_a=1.1,
                  truth_rank=32, truth_var=32 ** -0.5, noise_var=0.5),
    ),
}


def sweep_workloads():
    """The staleness / worker-count sweep on the mid data."""
    base = WORKLOADS["mid"]
    out = []
    for model in ("ssp", "essp"):
        for s in (0, 1, 2, 4, 8):
            for P in (1, 8, 64, 512):
                out.append(base.with_(name=f"sweep_{model}_s{s}_P{P}", model=model, s=s, P=P, clocks=20))
    return out


def workload(name: str) -> Workload:
    return WORKLOADS[name]
