"""The bench's gpu_launches figure is Iteration.launches_per_step(): a count of this
library's kernels per DBW iteration, written from the plan's rules (which GEMMs run
in three tf32 passes, which take the skinny kernels, which split K...).  Here the
kernels one iteration actually launches are counted from the CUDA activity record of
torch.profiler and compared with it, on every form of the pass."""
import pytest
import torch

from paper_2004_14696_gb300 import workloads
from paper_2004_14696_gb300.pipeline import Iteration

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)
    # the first profiling session of a process sets up the activity record: run one first
    try:
        with torch.profiler.profile(activities=[torch.profiler.ProfilerActivity.CUDA]):
            torch.zeros(16, device="cuda").add_(1)
            torch.cuda.synchronize()
    except RuntimeError:
        pass


def _wl(key, widths, n, B, prec, seed_offset):
    return workloads.Workload(key=key, widths=widths, n=n, B=B, prec=prec, S=900, feature_dist="normal",
                              time_model="shifted_exp", time_params={"shift": 1.0, "rate": 1.0}, lr=0.01,
                              seed_offset=seed_offset)


FP32, BF16 = workloads.PREC_FP32, workloads.PREC_BF16
CASES = [
    ("softmax784", workloads.SOFTMAX784, {"static_b": 4}),
    ("mlp784", workloads.MLP784, {}),
    # 3xTF32 forward (layer 1, with the gather's parts) and dW of layers 1 and 2
    ("tf32", _wl("lc_tf32", (516, 200, 136, 12), 21, 96, FP32, 101), {}),
    # fp32 shapes on the SIMT kernel with split K, and a one-layer model
    ("simt", _wl("lc_simt", (132, 200, 70, 7), 5, 3, FP32, 102), {}),
    ("linear", _wl("lc_linear", (132, 7), 5, 3, FP32, 103), {}),
    ("bf16", _wl("lc_bf16", (256, 128, 64, 10), 8, 32, BF16, 104), {}),
    ("bf16_simt", _wl("lc_bf16_simt", (200, 96, 10), 6, 16, BF16, 105), {}),
    ("received", _wl("lc_rx", (256, 128, 64, 10), 8, 32, BF16, 106), {"received": True}),
    ("psw", _wl("lc_psw", (256, 128, 64, 10), 8, 32, BF16, 107), {"clock": "psw"}),
]


def _our_kernels(prof):
    """Kernel launches of libdbw (every kernel of the library lives in namespace dbw)."""
    names = [e.name for e in prof.events() if e.device_type == torch.autograd.DeviceType.CUDA]
    return [nm for nm in names if "dbw::" in nm]


@pytest.mark.parametrize("name,wl,kw", CASES, ids=[c[0] for c in CASES])
def test_launches_per_step_matches_the_kernels_launched(name, wl, kw):
    it = Iteration(wl, **kw)
    for t in range(3):                  # the estimator starts choosing b at t = 2
        it.load_inputs(t)
        it.step()
    torch.cuda.synchronize()
    it.load_inputs(3)
    torch.cuda.synchronize()
    try:
        with torch.profiler.profile(activities=[torch.profiler.ProfilerActivity.CUDA]) as prof:
            it.step()
            torch.cuda.synchronize()
    except RuntimeError as e:           # no CUDA activity record on this host
        pytest.skip(f"torch.profiler CUDA activities unavailable: {e}")
    launched = _our_kernels(prof)
    if not launched:
        pytest.skip("torch.profiler recorded no kernel names")
    assert len(launched) == it.launches_per_step(), (len(launched), it.launches_per_step(), launched)
