"""The benchmark's byte model of the table algorithm (the roofline's
numerator) on trees whose counts are known by hand.  CPU only: it uses the
library's host-side row plan and no GPU."""
import numpy as np
import pytest

pytest.importorskip("torch")


@pytest.fixture(scope="module")
def bench():
    from paper_2608_01655_gb300 import build
    build.build()
    import bench as b
    return b


def _expect(n, k, pushes, internal):
    bmin = n * (k + 1) / 8 + 16 * n + 16 * (k + 1) * pushes + 8 * n
    return bmin, bmin + 8 * (k + 1) * internal


def test_chain(bench):
    """A chain: every skip row is the zero row (nothing pushed); every node
    but the leaf is internal."""
    n, k = 50, 16
    parent = np.arange(-1, n - 1, dtype=np.int32)
    t = bench.table_bytes(parent, k)
    assert (t["n_push"], t["n_internal"]) == (0, n - 1)
    assert (t["bmin_bytes_per_dp"], t["bstream_bytes_per_dp"]) == _expect(n, k, 0, n - 1)


def test_star_forest(bench):
    """Top-level chunks only: every skip row is the row just computed."""
    n, k = 40, 8
    t = bench.table_bytes(np.full(n, -1, np.int32), k)
    assert (t["n_push"], t["n_internal"]) == (0, 0)
    assert t["bmin_bytes_per_dp"] == _expect(n, k, 0, 0)[0]


def test_comb(bench):
    """A spine whose nodes each have a leaf as their last child (ids after the
    next spine node): a spine node's continuation, the row of its parent's
    leaf, is read after the whole subtree below it, so it is pushed; the root's
    continuation is the zero boundary row, so d spine nodes with children push
    d - 1 rows."""
    d = 12
    parent = [-1]
    spine = 0
    for _ in range(d):
        nxt = len(parent)
        parent.append(spine)            # the next spine node (smaller id: visited first)
        parent.append(spine)            # a leaf, the last child
        spine = nxt
    parent = np.asarray(parent, np.int32)
    n, k = len(parent), 32
    t = bench.table_bytes(parent, k)
    assert t["n_internal"] == d         # the spine nodes with children
    assert t["n_push"] == d - 1
    assert (t["bmin_bytes_per_dp"], t["bstream_bytes_per_dp"]) == _expect(n, k, d - 1, d)
