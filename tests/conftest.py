import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device and the built libdbw")


@pytest.fixture(scope="session")
def golden_dir():
    return os.path.join(ROOT, "tests", "golden")


def pytest_terminal_summary(terminalreporter):
    """What the bf16 acceptance rules took in this session: per test, the largest share
    of a worker's ReLU decisions taken from the GPU (R13) in any hidden layer, and the
    most entries beyond 2e-2 of their error scale in one compared row or vector."""
    try:
        import gpu_util
    except ImportError:
        return
    recs = gpu_util.ACCEPTANCE
    if not recs:
        return
    tr = terminalreporter
    tr.section("bf16 / ReLU acceptance taken")
    by = {}
    for r in recs:
        by.setdefault(r["test"], []).append(r)
    for test in sorted(by):
        rs = by[test]
        relu = [r for r in rs if r["kind"] == "relu"]
        outl = [r for r in rs if r["kind"] == "outliers"]
        parts = [r["text"] for r in rs if r["kind"] == "sampled"]
        if relu:
            frac = max(c / max(sz, 1) for r in relu for c, sz in zip(r["flips"], r["decisions"]))
            most = max(max(r["flips"]) if r["flips"] else 0 for r in relu)
            parts.append("relu: %d workers, max %d flips in a layer (%.2e of its decisions)" % (len(relu), most, frac))
        if outl:
            worst = max(outl, key=lambda r: r["outliers"] / max(r["entries"], 1))
            parts.append("outliers: max %d of %d entries (%.2e), worst ratio %.3g" % (
                worst["outliers"], worst["entries"], worst["outliers"] / max(worst["entries"], 1),
                max(r["worst"] for r in outl)))
        tr.write_line("%s: %s" % (test.split("::", 1)[-1], "; ".join(parts)))
