"""GPU test of dbw_aggregate_update_noalloc, the aggregation entry point for
callers that cannot allocate device memory (a plugin whose host application owns
the GPU memory budget, a loop that cannot afford cudaMalloc's synchronisation).

It must give the same result as dbw_aggregate_update with caller-provided
scratch, on two calls in a row (the built-in scratch array keeps the previous
call's contents, which must not leak into the next result), and must refuse a
size its fixed scratch cannot hold.  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

from paper_2004_14696_gb300 import dbw
from paper_2004_14696_gb300.pipeline import agg_case
from gpu_util import RTOL_FP32, assert_close_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _dev(x):
    return torch.as_tensor(np.ascontiguousarray(x)).cuda()


def _with_caller_scratch(G, w, mask, n, d, lr):
    """The existing path: dbw_aggregate_update into caller partials, totals via dbw_grad_stats."""
    wd = _dev(w)
    gb = torch.empty(d, dtype=torch.float32, device="cuda")
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    dbw.dbw_aggregate_update(_dev(G), n, d, mask, lr, wd, part, gb)
    state = dbw.new_state(n, 5)
    stats = torch.empty(dbw.STATS_LEN, dtype=torch.float64, device="cuda")
    rn = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_grad_stats(part, n, mask, torch.zeros(n, dtype=torch.float32, device="cuda"),
                       torch.arange(n, dtype=torch.float64, device="cuda"), lr, state, stats, rn)
    torch.cuda.synchronize()
    return wd.cpu().numpy(), gb.cpu().numpy(), stats.cpu().numpy(), rn.cpu().numpy()


def _select(n, times, b):
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    dbw.dbw_select_fastest(_dev(times), _dev(np.int32([b])), torch.empty(n, dtype=torch.int32, device="cuda"),
                           mask, torch.empty(n, dtype=torch.float64, device="cuda"))
    return mask


def test_noalloc_matches_caller_scratch_path_on_two_calls_in_a_row():
    lr = 0.05
    cases = [(64, 200003, 16), (16, 4097, 3)]      # the second call is smaller: stale scratch would show
    for (n, d, b) in cases:
        G, w, times = agg_case(n, d, seed=31 + n, b=b, mean=0.2)
        mask = _select(n, times, b)
        w_ref, g_ref, stats, rn = _with_caller_scratch(G, w, mask, n, d, lr)
        wd = _dev(w)
        gb = torch.empty(d, dtype=torch.float32, device="cuda")
        sums = torch.full((n + 2,), float("nan"), dtype=torch.float64, device="cuda")
        dbw.dbw_aggregate_update_noalloc(_dev(G), n, d, mask, lr, wd, sums, gb)
        torch.cuda.synchronize()
        s = sums.cpu().numpy()
        assert_close_rows(wd.cpu().numpy(), w_ref, RTOL_FP32, "w")
        assert_close_rows(gb.cpu().numpy(), g_ref, RTOL_FP32, "g_t")
        assert abs(s[n] - stats[dbw.STAT_SS]) <= RTOL_FP32 * abs(stats[dbw.STAT_SS])
        assert abs(s[n + 1] - stats[dbw.STAT_GBAR_SQ]) <= RTOL_FP32 * abs(stats[dbw.STAT_GBAR_SQ])
        m = mask.cpu().numpy().astype(bool)
        assert_close_rows(s[:n][m], rn[m], RTOL_FP32, "row norms")
        assert np.all(s[:n][~m] == 0.0)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    n = dbw.NMAX + 1
    G = torch.zeros((4, 8), dtype=torch.float32, device="cuda")
    with pytest.raises(dbw.DbwError) as e:
        dbw.dbw_aggregate_update_noalloc(G, n, 8, torch.ones(4, dtype=torch.uint8, device="cuda"), 0.1,
                                         torch.zeros(8, device="cuda"), torch.zeros(n + 2, dtype=torch.float64,
                                                                                     device="cuda"))
    assert e.value.code == dbw.DBW_EINVAL
