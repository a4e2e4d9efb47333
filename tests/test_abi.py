"""CPU checks of the C ABI: libdbw builds and loads without a GPU, exports every
entry point include/dbw.h declares, the Python mirror of dbw_state matches the C
layout, and host-side argument validation rejects bad calls before any launch."""
import ctypes as C
import os
import re
import subprocess

import pytest

from paper_2004_14696_gb300 import build as B
from paper_2004_14696_gb300 import dbw

HEADER = os.path.join(B.INCLUDE, "dbw.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return dbw.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(dbw_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 10
    for name in names:
        assert hasattr(lib, name), f"{name} declared in dbw.h but not exported"
    assert set(dbw.exported_symbols()) == set(names)


def test_state_layout_matches_c(tmp_path):
    fields = [f[0] for f in dbw.DbwState._fields_]
    src = tmp_path / "probe.c"
    body = "\n".join(f'printf("{f} %zu\\n", offsetof(dbw_state, {f}));' for f in fields)
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "dbw.h"\nint main(void){\n'
                   f'printf("sizeof %zu\\n", sizeof(dbw_state));\n{body}\nreturn 0;}}\n')
    exe = tmp_path / "probe"
    subprocess.run(["gcc", "-std=c99", "-I", B.INCLUDE, str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    got = dict(line.split() for line in out if line)
    assert int(got["sizeof"]) == C.sizeof(dbw.DbwState)
    for f in fields:
        assert int(got[f]) == getattr(dbw.DbwState, f).offset, f


def test_psw_header_layout_matches_c(tmp_path):
    fields = [f[0] for f in dbw.PswHeader._fields_]
    src = tmp_path / "probe_psw.c"
    body = "\n".join(f'printf("{f} %zu\\n", offsetof(dbw_psw_header, {f}));' for f in fields)
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "dbw.h"\nint main(void){\n'
                   f'printf("sizeof %zu\\n", sizeof(dbw_psw_header));\n{body}\nreturn 0;}}\n')
    exe = tmp_path / "probe_psw"
    subprocess.run(["gcc", "-std=c99", "-I", B.INCLUDE, str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    got = dict(line.split() for line in out if line)
    assert int(got["sizeof"]) == C.sizeof(dbw.PswHeader)
    for f in fields:
        assert int(got[f]) == getattr(dbw.PswHeader, f).offset, f
    assert dbw.dbw_psw_bytes(16) > 0 and dbw.dbw_psw_bytes(0) == 0 and dbw.dbw_psw_bytes(dbw.NMAX + 1) == 0


def test_param_count_and_workspace_queries(lib):
    assert dbw.dbw_param_count([784, 10]) == 7850
    assert dbw.dbw_param_count([4096, 4096, 4096, 4096, 1000]) == 54440936
    L, arr = dbw._widths([784, 0, 10])
    assert lib.dbw_param_count(L, arr) == -1
    ws32 = dbw.dbw_worker_grads_workspace_bytes([784, 256, 10], 64, 64, dbw.PREC_FP32)
    ws16 = dbw.dbw_worker_grads_workspace_bytes([784, 256, 10], 64, 64, dbw.PREC_BF16)
    assert ws32 > 0 and ws16 > 0 and ws16 < ws32 + 203530 * 2 + 4096
    assert dbw.dbw_worker_grads_workspace_bytes([784, 10], 0, 64, 0) == 0
    assert dbw.dbw_worker_grads_workspace_bytes([784, 10], 16, 32, 7) == 0


def test_host_validation_rejects_before_launch(lib):
    null = None
    # NULL pointers and out-of-range sizes are caught on the host (no device needed)
    assert lib.dbw_select_fastest(null, 4, null, null, null, null, null, null) == dbw.DBW_EINVAL
    assert b"NULL" in lib.dbw_last_error_string()
    assert lib.dbw_select_fastest(16, 0, 16, 16, 16, 16, null, null) == dbw.DBW_EINVAL
    assert lib.dbw_select_fastest(16, dbw.NMAX + 1, 16, 16, 16, 16, null, null) == dbw.DBW_EINVAL
    assert lib.dbw_aggregate_update(256, 6, 4, 5, 256, C.c_float(0.1), 256, null, 0, 256, 1 << 20,
                                    null) == dbw.DBW_EALIGN
    assert lib.dbw_aggregate_update(260, 8, 4, 5, 256, C.c_float(0.1), 256, null, 0, 256, 1 << 20,
                                    null) == dbw.DBW_EALIGN
    assert lib.dbw_aggregate_update(256, 8, 0, 5, 256, C.c_float(0.1), 256, null, 0, 256, 1 << 20,
                                    null) == dbw.DBW_EINVAL
    # an unknown flag bit is refused, for both aggregation entry points
    assert lib.dbw_aggregate_update(256, 8, 4, 5, 256, C.c_float(0.1), 256, null, 2, 256, 1 << 20,
                                    null) == dbw.DBW_EINVAL
    assert b"flags" in lib.dbw_last_error_string()
    assert lib.dbw_aggregate_update_noalloc(256, 8, 4, 5, 256, C.c_float(0.1), 256, null, 6, 256,
                                            null) == dbw.DBW_EINVAL
    # every entry point starts from an empty error text
    assert lib.dbw_param_count(1, null) == -1
    assert lib.dbw_aggregate_update_noalloc(256, 8, dbw.NMAX + 1, 5, 256, C.c_float(0.1), 256, null, 0, 256,
                                            null) == dbw.DBW_EINVAL
    assert lib.dbw_last_error_string() != b""
    assert lib.dbw_aggregate_update_noalloc(256, 6, 4, 5, 256, C.c_float(0.1), 256, null, 0, 256,
                                            null) == dbw.DBW_EALIGN
    assert b"ld" in lib.dbw_last_error_string() and b"n must" not in lib.dbw_last_error_string()
    assert lib.dbw_state_init(256, 4, 0, null) == dbw.DBW_EINVAL
    assert lib.dbw_state_init(256, 4, dbw.DMAX + 1, null) == dbw.DBW_EINVAL
    assert lib.dbw_choose_b(256, C.c_double(0.1), C.c_double(0.5), 0, 256, null, null) == dbw.DBW_EINVAL
    assert lib.dbw_choose_b(256, C.c_double(0.1), C.c_double(1.01), 4, 256, null, null) == dbw.DBW_EINVAL
    assert lib.dbw_grad_stats(256, 4, 256, 256, 256, C.c_double(-1.0), 256, null, null, null) == dbw.DBW_EINVAL
    L, arr = dbw._widths([784, 10])
    assert lib.dbw_worker_grads(L, arr, 0, 256, 7850, 256, 10, 256, 256, 16, 32, 256, 7850, 256, 256, 1 << 20,
                                null) == dbw.DBW_EALIGN   # ld % 4 != 0


def test_received_form_queries(lib):
    """The received-workers form: workspace only for the shapes it supports (bf16,
    B % 32 == 0, B | 128 or 128 | B), at least the per-worker pass's workspace (it
    extends that layout); a partials buffer of one block per quantity; host checks."""
    widths = [4096, 4096, 4096, 4096, 1000]
    full = dbw.dbw_worker_grads_workspace_bytes(widths, 256, 32, dbw.PREC_BF16)
    rx = dbw.dbw_received_grads_workspace_bytes(widths, 256, 32, dbw.PREC_BF16)
    assert rx > full > 0
    for n, B in ((128, 128), (4, 256), (8, 64)):
        assert dbw.dbw_received_grads_workspace_bytes([3072, 1024, 1024, 10], n, B, dbw.PREC_BF16) > 0
    assert dbw.dbw_received_grads_workspace_bytes(widths, 256, 32, dbw.PREC_FP32) == 0
    assert dbw.dbw_received_grads_workspace_bytes(widths, 256, 96, dbw.PREC_BF16) == 0
    assert dbw.dbw_received_grads_workspace_bytes(widths, 256, 16, dbw.PREC_BF16) == 0
    assert dbw.dbw_received_partials_bytes(16) == 8 * (4 + 2 * 18)
    assert dbw.dbw_received_partials_bytes(0) == 0 and dbw.dbw_received_partials_bytes(dbw.NMAX + 1) == 0
    L, arr = dbw._widths([784, 10])
    null = None
    args = [L, arr, dbw.PREC_BF16, 256, 7850, 256, 10, 256, 256, 16, 32, 256, C.c_float(0.1), null, 256, 256]
    assert lib.dbw_received_grads_update(*args, 1 << 20, 256, 1 << 30, null) != dbw.DBW_OK   # no device here
    assert lib.dbw_received_grads_update(*args[:3], null, *args[4:], 1 << 20, 256, 1 << 30, null) == dbw.DBW_EINVAL
    assert lib.dbw_received_grads_update(*args, 16, 256, 1 << 30, null) == dbw.DBW_EINVAL          # partials too small
    args[3] = 260
    assert lib.dbw_received_grads_update(*args, 1 << 20, 256, 1 << 30, null) == dbw.DBW_EALIGN
