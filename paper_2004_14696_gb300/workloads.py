"""The five synthetic workloads the DBW iteration is checked and measured on.

Shapes follow the paper's experiments (Sect. 4): MNIST-like 784-feature /
10-class data, CIFAR-like 3072 features, n workers each with a minibatch of B
samples, round-trip times from the shifted-exponential / heavy-tailed families,
the window D = 5 and the loss-increase factor beta = 1.01 (Sect. 3.3).  The
datasets themselves are replaced by seeded synthetic pools (see ``inputs``).
"""
from __future__ import annotations

from dataclasses import dataclass, field

from . import inputs

PREC_FP32 = 0
PREC_BF16 = 1


@dataclass(frozen=True)
class Workload:
    key: str
    widths: tuple            # layer widths, input first, classes last
    n: int                   # workers
    B: int                   # minibatch per worker
    prec: int                # PREC_FP32 or PREC_BF16 (GEMM operand type)
    S: int                   # samples in the synthetic pool
    feature_dist: str        # "normal" or "uniform"
    time_model: str
    time_params: dict = field(default_factory=dict)
    iters: int = 100
    lr: float = 0.05
    D: int = 5
    beta: float = 1.01
    policy: str = "dbw"      # "dbw" (choose b every iteration) or "static"
    seed_offset: int = 0
    # learning rate of static-b runs: "fixed" (lr for every k) or "proportional"
    # (lr * k / n, the rule Sect. 4 uses for static settings); DBW always uses lr
    lr_rule: str = "fixed"

    def lr_for(self, k: int) -> float:
        """Learning rate of an iteration that keeps k gradients (static-b runs)."""
        if self.lr_rule == "proportional":
            return self.lr * k / self.n
        return self.lr

    @property
    def seed(self) -> int:
        return inputs.BASE_SEED + self.seed_offset

    @property
    def d(self) -> int:
        return inputs.param_count(self.widths)

    @property
    def ld(self) -> int:
        # rows of G start on 128-byte boundaries (the weight-gradient kernel writes
        # whole 32-byte sectors with 256-bit stores when rows are 32-byte aligned)
        return inputs.round_up(self.d, 32)

    @property
    def classes(self) -> int:
        return int(self.widths[-1])

    @property
    def M(self) -> int:
        return self.n * self.B


SOFTMAX784 = Workload(
    key="softmax784_n16_B32", widths=(784, 10), n=16, B=32, prec=PREC_FP32,
    S=60000, feature_dist="normal", time_model="shifted_exp",
    time_params={"shift": 1.0, "rate": 1.0}, iters=100, lr=0.05,
    policy="static", seed_offset=1)

MLP784 = Workload(
    key="mlp784-256-10_n64_B64", widths=(784, 256, 10), n=64, B=64,
    prec=PREC_FP32, S=60000, feature_dist="normal", time_model="lognormal",
    time_params={"mu": 0.0, "sigma": 0.5}, iters=200, lr=0.05, seed_offset=2)

MLP3072 = Workload(
    key="mlp3072-1024-1024-10_n128_B128", widths=(3072, 1024, 1024, 10), n=128,
    B=128, prec=PREC_BF16, S=50000, feature_dist="uniform",
    time_model="exp_slow", time_params={"rate": 1.0, "frac": 0.05, "factor": 10.0},
    iters=200, lr=0.01, seed_offset=4)

MLP4096 = Workload(
    key="mlp4096x3-1000_n256_B32", widths=(4096, 4096, 4096, 4096, 1000), n=256,
    B=32, prec=PREC_BF16, S=32768, feature_dist="normal", time_model="pareto",
    time_params={"alpha": 2.0, "xm": 1.0}, iters=200, lr=0.01, seed_offset=5)

# Aggregation-only sweep: G ~ N(0,1) [n, d], exponential times, b in {0, n/4}.
AGG_NS = (16, 64, 256)
AGG_DS = (10**5, 10**6, 10**7, 10**8)
AGG_SEED = inputs.BASE_SEED + 3
AGG_MAX_BYTES = 180 * 10**9

ALL = {w.key: w for w in (SOFTMAX784, MLP784, MLP3072, MLP4096)}
