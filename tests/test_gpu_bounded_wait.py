"""GPU test of the bounded-wait path of the tensor-core kernels.

Every wait of a tensor-core kernel on a pipeline barrier is bounded.  When one runs
out the kernel raises bit 0 of the status word, stops, waits (bounded) for its own
copies still in flight, releases its tensor memory and returns.  The test makes one
wait run out without faulting anything: dbw_test_arm_wait_timeout keeps the first
CTA of the next weight-gradient launch from issuing one stage's TMA load (no copy is
then outstanding for that stage) and shortens the bound to 1 ms.  Then: the call
returns, the status word has bit 0 set, and the next normal call on the same process
(which allocates the same tensor memory again) gives the oracle's result.  A tiny
shape only."""
import numpy as np
import pytest
import torch

from oracle import dbw_oracle as O
from paper_2004_14696_gb300 import dbw, workloads
from paper_2004_14696_gb300.pipeline import Iteration
from gpu_util import RTOL_BF16, assert_worker_grads_match, gpu_active_sets

pytestmark = pytest.mark.gpu

TINY = workloads.Workload(key="wait_tiny", widths=(64, 32, 10), n=2, B=32, prec=workloads.PREC_BF16, S=200,
                          feature_dist="normal", time_model="shifted_exp", time_params={"shift": 1.0, "rate": 1.0},
                          lr=0.01, seed_offset=97)


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _grads(it):
    wl = it.wl
    dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.G, it.loss, it.ws)
    torch.cuda.synchronize()
    return int(it.ws[:4].view(torch.int32).item())


def test_a_wait_that_runs_out_sets_the_status_and_the_next_call_is_exact():
    wl = TINY
    it = Iteration(wl, static_b=0)
    it.load_inputs(0)
    assert _grads(it) == 0
    dbw.dbw_test_arm_wait_timeout(0, 1.0)
    assert _grads(it) & 1, "the wait for the stage without its load did not run out"
    # armed once: the next call is a normal one, on the same process and tensor memory
    assert _grads(it) == 0
    w = it.w.cpu().numpy().astype(np.float64)
    idx, _ = it.host_inputs(0)
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    assert_worker_grads_match(it.G.cpu().numpy()[:, :wl.d], it.loss.cpu().numpy(), wl.widths, w, pool[idx],
                              labels[idx], wl.B, True, range(wl.n), RTOL_BF16,
                              gpu_active=gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec))


def test_arming_is_checked_and_can_be_undone():
    with pytest.raises(dbw.DbwError):
        dbw.dbw_test_arm_wait_timeout(0, 0.0)
    with pytest.raises(dbw.DbwError):
        dbw.dbw_test_arm_wait_timeout(0, 5000.0)
    dbw.dbw_test_arm_wait_timeout(0, 1.0)
    dbw.dbw_test_arm_wait_timeout(-1, 0.0)          # disarmed: the next call runs normally
    it = Iteration(TINY, static_b=0)
    it.load_inputs(0)
    assert _grads(it) == 0
