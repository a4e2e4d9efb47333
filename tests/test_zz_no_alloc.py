"""GPU test of dbw_aggregate_update_noalloc, the aggregation entry point for
callers that cannot allocate device memory (a plugin whose host application owns
the GPU memory budget, a loop that cannot afford cudaMalloc's synchronisation).

It must give the same result as dbw_aggregate_update with caller-provided
scratch, and the oracle's, on two calls in a row (the built-in scratch array
keeps the previous call's contents, which must not leak into the next result);
its fixed scratch must cover every n the library accepts on this device; and a
refused call must not leave its message behind for the next successful one.
This file is collected last on purpose."""
import numpy as np
import pytest
import torch

from oracle import dbw_oracle as O
from paper_2004_14696_gb300 import dbw
from paper_2004_14696_gb300.pipeline import agg_case
from gpu_util import RTOL_FP32, assert_close_rows, assert_close_scalar

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _dev(x):
    return torch.as_tensor(np.ascontiguousarray(x)).cuda()


def _with_caller_scratch(G, w, mask, n, d, lr, flags):
    """The existing path: dbw_aggregate_update into caller partials, totals via dbw_grad_stats."""
    wd = _dev(w)
    gb = torch.empty(d, dtype=torch.float32, device="cuda")
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    dbw.dbw_aggregate_update(_dev(G), n, d, mask, lr, wd, part, gb, flags=flags)
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


@pytest.mark.parametrize("flags", [0, dbw.ALL_ROW_NORMS])
def test_noalloc_matches_caller_scratch_path_and_oracle_on_two_calls_in_a_row(flags):
    lr = 0.05
    cases = [(64, 200003, 16), (16, 4097, 3)]      # the second call is smaller: stale scratch would show
    for (n, d, b) in cases:
        G, w, times = agg_case(n, d, seed=31 + n, b=b, mean=0.2)
        mask = _select(n, times, b)
        w_ref, g_ref, stats, rn = _with_caller_scratch(G, w, mask, n, d, lr, flags)
        wd = _dev(w)
        gb = torch.empty(d, dtype=torch.float32, device="cuda")
        sums = torch.full((n + 2,), float("nan"), dtype=torch.float64, device="cuda")
        dbw.dbw_aggregate_update_noalloc(_dev(G), n, d, mask, lr, wd, sums, gb, flags=flags)
        torch.cuda.synchronize()
        assert dbw.lib().dbw_last_error_string() == b""
        s = sums.cpu().numpy()
        # against the call with caller scratch: the same kernel and reduction order
        assert np.array_equal(wd.cpu().numpy(), w_ref) and np.array_equal(gb.cpu().numpy(), g_ref)
        assert s[n] == stats[dbw.STAT_SS] and s[n + 1] == stats[dbw.STAT_GBAR_SQ]
        m = mask.cpu().numpy().astype(bool)
        assert np.array_equal(s[:n][m], rn[m])
        # against the oracle
        _, mo, _ = O.select_fastest(times, b)
        assert np.array_equal(mo.astype(bool), m)
        Gd = G[:, :d]
        gbar = O.aggregate(Gd, mo)
        assert_close_rows(gb.cpu().numpy(), gbar, RTOL_FP32, "g_t")
        assert_close_rows(wd.cpu().numpy(), O.sgd_update(w, gbar, lr), RTOL_FP32, "w_{t+1}")
        assert_close_scalar(s[n], O.deviation_sumsq(Gd, mo, gbar), RTOL_FP32, "deviation sum of Eq. (10)")
        assert_close_scalar(s[n + 1], float(gbar @ gbar), RTOL_FP32, "||g_t||^2")
        r = O.row_sqnorms(Gd, mo, all_rows=bool(flags))
        if flags:
            assert_close_rows(s[:n], r, RTOL_FP32, "every row's squared norm")
        else:
            assert_close_rows(s[:n][m], r[m], RTOL_FP32, "received rows' squared norms")
            assert np.all(s[:n][~m] == 0.0)


def test_noalloc_scratch_covers_every_n_on_this_device():
    """The built-in array is large enough for every n the library accepts (the
    partials grow with n and with the aggregation's grid, SMs x resident blocks)."""
    need = [dbw.dbw_aggregate_partials_bytes(n, 10 ** 8) for n in range(1, dbw.NMAX + 1)]
    assert min(need) > 0
    assert max(need) <= dbw.NOALLOC_SCRATCH_BYTES, (max(need), int(np.argmax(need)) + 1)


def test_noalloc_n_range_check_and_error_text_cleared():
    """n beyond DBW_NMAX is refused by the n-range check before any launch; the next
    successful call leaves no error text behind."""
    n = dbw.NMAX + 1
    G = torch.zeros((4, 8), dtype=torch.float32, device="cuda")
    with pytest.raises(dbw.DbwError) as e:
        dbw.dbw_aggregate_update_noalloc(G, n, 8, torch.ones(4, dtype=torch.uint8, device="cuda"), 0.1,
                                         torch.zeros(8, device="cuda"), torch.zeros(n + 2, dtype=torch.float64,
                                                                                     device="cuda"))
    assert e.value.code == dbw.DBW_EINVAL
    assert dbw.lib().dbw_last_error_string() != b""
    sums = torch.zeros(6, dtype=torch.float64, device="cuda")
    dbw.dbw_aggregate_update_noalloc(G, 4, 8, torch.ones(4, dtype=torch.uint8, device="cuda"), 0.1,
                                     torch.zeros(8, device="cuda"), sums)
    torch.cuda.synchronize()
    assert dbw.lib().dbw_last_error_string() == b""
    assert np.all(sums.cpu().numpy() == 0.0)
