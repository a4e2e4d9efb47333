"""GPU parity of the received-workers form of the iteration (dbw_received_grads_update):
Eqs. (2)-(4) and the statistics of Sect. 3.1 for the k received workers, without
the [n, d] gradient matrix.  Against the oracle on small workloads (every output),
on the full-size bf16 workloads on sampled workers, and through the edge cases
(k = n, k = 1, empty mask, poisoned samples, unsupported shapes)."""
import math
import os

import numpy as np
import pytest
import torch

from oracle import dbw_oracle as O
from paper_2004_14696_gb300 import dbw, inputs, workloads
from paper_2004_14696_gb300.pipeline import Iteration
from gpu_util import (RTOL_BF16, assert_bf16_close, assert_close_scalar, assert_close_to_magnitude,
                      gpu_active_sets, oracle_rows_with_decisions, param_blocks, tensor_scale)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _wl(key, widths, n, B, seed_offset, dist="normal"):
    return workloads.Workload(key=key, widths=widths, n=n, B=B, prec=workloads.PREC_BF16, S=600,
                              feature_dist=dist, time_model="exp_slow",
                              time_params={"rate": 1.0, "frac": 0.25, "factor": 10.0}, lr=0.01,
                              seed_offset=seed_offset)


# B = 32: four workers per 128-row tile; B = 64 with widths that are not multiples of 8;
# B = 128: one worker per tile; B = 256: a worker spans 2 x 2 Gram tiles
RX_B32 = _wl("rx_b32", (256, 128, 64, 10), 8, 32, 91)
RX_B64 = _wl("rx_b64", (300, 200, 100, 7), 5, 64, 92, "uniform")
RX_B128 = _wl("rx_b128", (128, 96, 10), 3, 128, 93)
RX_B256 = _wl("rx_b256", (200, 64, 12), 3, 256, 94)
# k B long enough for the mean-gradient GEMM to split K over several work items (its
# outputs have far fewer tiles than SMs); b = 31 leaves one worker, so most splits are empty
RX_SPLIT = _wl("rx_split", (256, 96, 10), 32, 64, 96)
# a single worker (n = 1): one 32-row slot, k = 1
RX_ONE = _wl("rx_one", (512, 384, 10), 1, 32, 98)
# B (C + 8) bf16 larger than the softmax kernel's transposing tile: dZ_L^T by the separate
# transpose kernel
RX_WIDE = _wl("rx_wide", (64, 320), 3, 256, 99)


def slot_rows(mask, B):
    """rows_of for the received form: worker j = the s-th received worker sits at rows s*B .."""
    slot = {int(j): s for s, j in enumerate(np.flatnonzero(mask))}
    return lambda j: slice(slot[j] * B, (slot[j] + 1) * B)


def run_received(wl, b, t=0):
    it = Iteration(wl, static_b=b, keep_gbar=True, received=True)
    w0 = it.w.cpu().numpy().astype(np.float64)
    idx, times = it.host_inputs(t)
    it.load_inputs(t)
    it.step()
    torch.cuda.synchronize()
    assert int(it.ws[:4].view(torch.int32).item()) == 0, "device status word set"
    return it, w0, idx, times


def check_against_oracle(it, wl, w0, idx, times, b, workers=None):
    """Every received worker (or the sampled ``workers``): loss and ||g_j||^2 against
    the oracle's Eq. (2) row; with all of them, g_t, w_{t+1}, SS and ||g_t||^2."""
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    _, mask, ts = O.select_fastest(times, b)
    assert np.array_equal(it.mask.cpu().numpy(), mask)
    received = [int(j) for j in np.flatnonzero(mask)]
    k = len(received)
    blocks = param_blocks(wl.widths)
    active = gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec)
    check = received if workers is None else workers
    rows = oracle_rows_with_decisions(wl.widths, w0, pool[idx], labels[idx], wl.B, True, check, active,
                                      rows_of=slot_rows(mask, wl.B))
    loss = it.loss.cpu().numpy()
    rn = it.row_sqnorm.cpu().numpy()
    for j in range(wl.n):
        if mask[j]:
            if j in rows:
                assert_close_scalar(loss[j], rows[j][1], RTOL_BF16, f"loss of worker {j}")
                assert_close_scalar(rn[j], float(rows[j][0] @ rows[j][0]), RTOL_BF16, f"||g_{j}||^2")
        else:
            assert math.isnan(loss[j]) and math.isnan(rn[j]), f"worker {j} was not received"
    s = it.stats.cpu().numpy()
    assert s[dbw.STAT_K] == k
    if workers is not None:
        return
    G_ref = np.zeros((wl.n, wl.d))
    G_mag = np.zeros((wl.n, wl.d))
    loss_ref = np.zeros(wl.n)
    for j in received:
        G_ref[j], loss_ref[j] = rows[j][0], rows[j][1]
        G_mag[j] = np.maximum(rows[j][2], tensor_scale(rows[j][0], blocks))
    gbar = O.aggregate(G_ref, mask)
    mag = O.aggregate(G_mag, mask)
    assert_bf16_close(it.gbar.cpu().numpy(), gbar, mag, blocks, RTOL_BF16, "g_t")
    w_new = O.sgd_update(w0, gbar, wl.lr)
    assert_close_to_magnitude(it.w.cpu().numpy(), w_new, wl.lr * mag, RTOL_BF16, "w",
                              extra=2.0 ** -20 * np.abs(w_new))
    assert_close_scalar(s[dbw.STAT_GBAR_SQ], float(gbar @ gbar), RTOL_BF16, "||g_t||^2")
    assert_close_scalar(s[dbw.STAT_F], float(np.mean(loss_ref[received])), RTOL_BF16, "F")
    if k >= 2:
        # SS is formed as sum_j ||g_j||^2 - k ||g_t||^2: its error scale is the sum of the terms
        SS = O.deviation_sumsq(G_ref, mask, gbar)
        norms = sum(float(G_ref[j] @ G_ref[j]) for j in received)
        assert abs(s[dbw.STAT_SS] - SS) <= RTOL_BF16 * norms, (s[dbw.STAT_SS], SS, norms)
        assert s[dbw.STAT_SS] > 0


@pytest.mark.parametrize("wl,b", [(RX_B32, 0), (RX_B32, 3), (RX_B32, 7), (RX_B64, 0), (RX_B64, 2),
                                  (RX_B128, 1), (RX_B256, 0), (RX_B256, 2), (RX_SPLIT, 5), (RX_SPLIT, 31),
                                  (RX_ONE, 0), (RX_WIDE, 1)],
                         ids=lambda v: v.key if hasattr(v, "key") else f"b{v}")
def test_received_iteration_matches_oracle(wl, b):
    """All outputs of one received-workers iteration against the oracle: loss (NaN for
    the workers left out), ||g_j||^2 of every received worker, g_t, w_{t+1}, ||g_t||^2,
    F^_t and the deviation sum; b = n - 1 keeps a single worker."""
    it, w0, idx, times = run_received(wl, b)
    check_against_oracle(it, wl, w0, idx, times, b)


def test_received_deterministic():
    """Fixed-order reductions everywhere: two runs give identical bits."""
    a, *_ = run_received(RX_B32, 2)
    c, *_ = run_received(RX_B32, 2)
    assert torch.equal(a.w, c.w) and torch.equal(a.gbar, c.gbar)
    # bit patterns (L^+ is NaN at t = 0, and NaN != NaN)
    assert torch.equal(a.stats.view(torch.int64), c.stats.view(torch.int64))
    assert torch.equal(a.partials, c.partials)


def test_received_dbw_trajectory_independent():
    """DBW iterations in the received form: GPU and oracle run their own trajectories
    from the same seeds; b_t agrees exactly unless the oracle's decision is within
    1e-3 of flipping (then the comparison stops)."""
    from test_gpu_parity import decision_margin
    wl = RX_B32
    it = Iteration(wl, keep_gbar=True, received=True)
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    ost = O.State(n=wl.n, D=wl.D)
    w_or = inputs.kaiming_uniform_params(wl.seed, wl.widths).astype(np.float64)
    blocks = param_blocks(wl.widths)
    compared = 0
    for t in range(8):
        idx, times = it.host_inputs(t)
        margin = decision_margin(ost, wl.lr, wl.beta)
        k_or, _ = O.choose_k(ost, wl.lr, wl.beta)
        it.load_inputs(t)
        it.step()
        torch.cuda.synchronize()
        b = int(it.b.item())
        if wl.n - b != k_or:
            assert margin < 1e-3, (t, b, k_or, margin)
            break
        order, mask, ts = O.select_fastest(times, b)
        assert np.array_equal(it.mask.cpu().numpy(), mask)
        received = [int(j) for j in np.flatnonzero(mask)]
        rows = oracle_rows_with_decisions(wl.widths, w_or, pool[idx], labels[idx], wl.B, True, received,
                                          gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec),
                                          rows_of=slot_rows(mask, wl.B))
        G_ref = np.zeros((wl.n, wl.d))
        G_mag = np.zeros((wl.n, wl.d))
        loss_ref = np.zeros(wl.n)
        for j in received:
            G_ref[j], loss_ref[j] = rows[j][0], rows[j][1]
            G_mag[j] = np.maximum(rows[j][2], tensor_scale(rows[j][0], blocks))
        gbar = O.aggregate(G_ref, mask)
        mag = O.aggregate(G_mag, mask)
        w_new = O.sgd_update(w_or, gbar, wl.lr)
        SS = O.deviation_sumsq(G_ref, mask, gbar)
        rec = O.record_iteration(ost, wl.n - b, SS, float(gbar @ gbar), loss_ref, mask, ts, wl.lr)
        assert_bf16_close(it.gbar.cpu().numpy(), gbar, mag, blocks, RTOL_BF16, f"g_t at t={t}")
        assert_close_to_magnitude(it.w.cpu().numpy(), w_new, wl.lr * mag, RTOL_BF16, "w",
                                  extra=2.0 ** -20 * np.abs(w_new))
        s = it.stats.cpu().numpy()
        assert_close_scalar(s[dbw.STAT_GBAR_SQ], rec["gbar_sq"], RTOL_BF16, "||g_t||^2")
        assert_close_scalar(s[dbw.STAT_F], rec["F"], RTOL_BF16, "F")
        assert s[dbw.STAT_VCLOCK] == rec["vclock"]
        w_or = w_new
        compared += 1
    assert compared >= 3


def sampled_entries(widths, seed, side=64):
    """Seeded side x side blocks of every layer's W and every bias, as indices into a
    row of G / into w; returns (entries, tensor index of each entry, the blocks' list,
    one [start, end) range of the entry list per sampled tensor)."""
    rng = np.random.default_rng(seed)
    blocks = param_blocks(widths)
    ent, ten, listed, ranges = [], [], [], []
    for l in range(len(widths) - 1):
        fin, fout = int(widths[l]), int(widths[l + 1])
        (a, _), (ab, bb) = blocks[2 * l], blocks[2 * l + 1]
        h, wd = min(side, fout), min(side, fin)
        r0, c0 = int(rng.integers(0, fout - h + 1)), int(rng.integers(0, fin - wd + 1))
        start = len(ent)
        for r in range(r0, r0 + h):
            ent.extend(range(a + r * fin + c0, a + r * fin + c0 + wd))
            ten.extend([2 * l] * wd)
        ranges.append((start, len(ent)))
        listed.append(f"W_{l + 1}[{r0}:{r0 + h}, {c0}:{c0 + wd}]")
        start = len(ent)
        ent.extend(range(ab, bb))
        ten.extend([2 * l + 1] * (bb - ab))
        ranges.append((start, len(ent)))
        listed.append(f"b_{l + 1}[0:{fout}]")
    return np.array(ent, dtype=np.int64), np.array(ten, dtype=np.int64), listed, ranges


@pytest.mark.parametrize("wl", [workloads.MLP3072, workloads.MLP4096], ids=lambda w: w.key)
def test_received_full_size_against_oracle(wl):
    """Full-size bf16 workloads with b = n/4 (k = 96 and 192 received workers), in the
    launch configuration the bench times, against the oracle's Eq. (2) row of EVERY
    received worker (formed in spawned processes; each worker's row depends only on its
    B samples, w and the GPU's certified-ambiguous ReLU decisions, R13): every received
    worker's loss and ||g_j||^2; g_t and w_{t+1} element by element on a seeded 64 x 64
    block of every layer's W and on every bias (R17); ||g_t||^2; the deviation sum of
    Eq. (10) against sum_j ||g_j||^2 - k ||g_t||^2 (the identity pinned in the oracle
    tests).  The mean over the k rows is summed as the rows are formed: the k full rows
    (83 GB in fp64 for k = 192) are never held at once, and each column's mean is
    independent of the others."""
    from gpu_util import ACCEPTANCE, oracle_rows_in_pool
    b = wl.n // 4
    it, w0, idx, times = run_received(wl, b)
    _, mask, _ = O.select_fastest(times, b)
    assert np.array_equal(it.mask.cpu().numpy(), mask)
    received = [int(j) for j in np.flatnonzero(mask)]
    k = len(received)
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    blocks = param_blocks(wl.widths)
    ent, ten, listed, ranges = sampled_entries(wl.widths, wl.seed + 17)
    active = gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec)     # rows in slot order
    procs = min(os.cpu_count() or 1, 16)
    chunks = [received[q::procs] for q in range(procs) if received[q::procs]]
    slot = {j: s for s, j in enumerate(received)}
    tasks = []
    for ch in chunks:
        rows = np.concatenate([np.arange(j * wl.B, (j + 1) * wl.B) for j in ch])
        srows = np.concatenate([np.arange(slot[j] * wl.B, (slot[j] + 1) * wl.B) for j in ch])
        tasks.append((pool[idx[rows]], labels[idx[rows]], wl.B, [a[srows] for a in active]))
    out = oracle_rows_in_pool(wl.widths, wl.seed, True, ent, ten, blocks, tasks)
    per = {}
    total = np.zeros(wl.d)
    for ch, (res, tot, _) in zip(chunks, out):
        total += tot
        for j, r in zip(ch, res):
            per[j] = r
    loss = it.loss.cpu().numpy()
    rn = it.row_sqnorm.cpu().numpy()
    for j in range(wl.n):
        if mask[j]:
            assert_close_scalar(loss[j], per[j][0], RTOL_BF16, f"loss of worker {j}")
            assert_close_scalar(rn[j], per[j][1], RTOL_BF16, f"||g_{j}||^2")
        else:
            assert math.isnan(loss[j]) and math.isnan(rn[j]), f"worker {j} was not received"
    G_ent = np.stack([per[j][2] for j in received])
    S_ent = np.stack([per[j][3] for j in received])
    ones = np.ones(k, dtype=np.uint8)
    gbar_ent = O.aggregate(G_ent, ones)
    mag_ent = O.aggregate(S_ent, ones)
    sub = [(a, b2) for (a, b2) in ranges]
    assert_bf16_close(it.gbar.cpu().numpy()[ent], gbar_ent, mag_ent, sub, RTOL_BF16, "g_t on the sampled entries")
    w_new = O.sgd_update(w0[ent], gbar_ent, wl.lr)
    assert_close_to_magnitude(it.w.cpu().numpy()[ent], w_new, wl.lr * mag_ent, RTOL_BF16,
                              "w_{t+1} on the sampled entries", extra=2.0 ** -20 * np.abs(w_new))
    gbar = total / k
    s = it.stats.cpu().numpy()
    g2 = float(gbar @ gbar)
    assert_close_scalar(s[dbw.STAT_GBAR_SQ], g2, RTOL_BF16, "||g_t||^2")
    norms = sum(per[j][1] for j in received)
    SS = norms - k * g2
    assert SS > 0 and s[dbw.STAT_SS] > 0
    assert abs(s[dbw.STAT_SS] - SS) <= RTOL_BF16 * norms, (s[dbw.STAT_SS], SS, norms)
    assert_close_scalar(s[dbw.STAT_F], float(np.mean([per[j][0] for j in received])), RTOL_BF16, "F")
    ACCEPTANCE.append({"test": os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0], "kind": "sampled",
                       "text": f"k = {k} workers against the oracle; g_t, w on " + ", ".join(listed)})


def test_received_empty_mask_changes_nothing():
    """k = 0 (a mask with no byte set): nothing is launched on any row, w is unchanged,
    every loss is NaN and the sums are NaN; dbw_grad_stats flags the empty mask."""
    wl = RX_B32
    it = Iteration(wl, static_b=0, keep_gbar=True, received=True)
    it.load_inputs(0)
    w_before = it.w.clone()
    it.mask.zero_()
    tsorted = torch.arange(1, wl.n + 1, dtype=torch.float64, device="cuda")
    dbw.dbw_received_grads_update(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.mask, wl.lr,
                                  it.loss, it.partials, it.ws, it.gbar)
    dbw.dbw_grad_stats(it.partials, wl.n, it.mask, it.loss, tsorted, wl.lr, it.state, it.stats)
    torch.cuda.synchronize()
    assert torch.equal(it.w, w_before)
    assert torch.isnan(it.loss).all()
    vals = it.partials.view(torch.float64)[4 + wl.n + 2:]
    assert torch.isnan(vals[wl.n:wl.n + 2]).all() and (vals[:wl.n] == 0).all()
    assert dbw.read_state(it.state).flags & dbw.FLAG_EMPTY_MASK


def test_received_poisoned_samples():
    """An out-of-range sample index of a received worker makes its loss NaN (and,
    through g_t, the update); one of a worker that is not received changes nothing:
    its gradient is never formed."""
    wl = RX_B32
    b = 3
    base, *_ = run_received(wl, b)
    _, mask, _ = O.select_fastest(base.times.cpu().numpy(), b)
    out_j = int(np.flatnonzero(mask == 0)[0])
    in_j = int(np.flatnonzero(mask)[0])

    it = Iteration(wl, static_b=b, keep_gbar=True, received=True)
    idx, _ = it.host_inputs(0)
    it.load_inputs(0)
    idx[out_j * wl.B + 5] = wl.S + 11
    it.idx.copy_(torch.from_numpy(idx))
    it.step()
    torch.cuda.synchronize()
    assert torch.equal(it.w, base.w) and torch.equal(it.stats.view(torch.int64), base.stats.view(torch.int64))

    it = Iteration(wl, static_b=b, keep_gbar=True, received=True)
    idx, _ = it.host_inputs(0)
    it.load_inputs(0)
    idx[in_j * wl.B + 2] = -4
    it.idx.copy_(torch.from_numpy(idx))
    it.step()
    torch.cuda.synchronize()
    loss = it.loss.cpu().numpy()
    assert math.isnan(loss[in_j])
    others = [j for j in np.flatnonzero(mask) if j != in_j]
    assert np.isfinite(loss[others]).all()


def test_received_unsupported_shapes_are_refused():
    """fp32 operands, B not a multiple of 32, and B = 96 (neither divides 128 nor is a
    multiple of it) are refused on the host with DBW_EUNSUPPORTED; nothing runs."""
    wl = RX_B32
    it = Iteration(wl, static_b=0, received=True)
    for prec, B in ((dbw.PREC_FP32, 32), (dbw.PREC_BF16, 16), (dbw.PREC_BF16, 96)):
        n = 4
        idx = torch.zeros(n * B, dtype=torch.int32, device="cuda")
        mask = torch.ones(n, dtype=torch.uint8, device="cuda")
        loss = torch.empty(n, dtype=torch.float32, device="cuda")
        part = torch.empty(dbw.dbw_received_partials_bytes(n), dtype=torch.uint8, device="cuda")
        assert dbw.dbw_received_grads_workspace_bytes(wl.widths, n, B, prec) == 0
        with pytest.raises(dbw.DbwError) as e:
            dbw.dbw_received_grads_update(wl.widths, prec, it.w, it.pool, it.labels, idx, n, B, mask, wl.lr, loss,
                                          part, it.ws)
        assert e.value.code == dbw.DBW_EUNSUPPORTED


def test_launch_timing_channels():
    """dbw_profile_gemm / dbw_profile_dw record one event pair per persistent GEMM and per
    weight-gradient launch, only while enabled; a read forgets the records."""
    L = len(RX_B32.widths) - 1
    # received form: L forward GEMMs, then per layer one launch of the mean-gradient GEMM
    # (with the dX GEMM of that layer when l > 0)
    for received, gemms, dws in ((False, L + (L - 1), L), (True, L + L, 0)):
        it = Iteration(RX_B32, static_b=2, received=received)
        it.load_inputs(0)
        it.step()
        torch.cuda.synchronize()
        dbw.dbw_profile_gemm(True)
        dbw.dbw_profile_dw(True)
        it.step()
        torch.cuda.synchronize()
        ms, launches = dbw.dbw_profile_gemm_read()
        dms, dl, dbytes = dbw.dbw_profile_dw_read()
        assert launches == gemms and ms > 0
        assert dl == dws and (dws == 0 or (dms > 0 and dbytes > 0))
        assert dbw.dbw_profile_gemm_read() == (0.0, 0)
        dbw.dbw_profile_gemm(False)
        dbw.dbw_profile_dw(False)
        it.step()
        torch.cuda.synchronize()
        assert dbw.dbw_profile_gemm_read() == (0.0, 0)
        assert dbw.dbw_profile_dw_read()[1] == 0
