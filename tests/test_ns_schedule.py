"""The persistent work tables, checked on the host.

The library builds the tables the persistent launches claim from with the
same code the GPU path uses (malt_ns_schedule needs no GPU).  The Orth step
of Algorithm 1 iterates A = X X^T, B' = aI + bA + cA^2, X <- B' X on each
matrix's own data, so for each table:
  * every tile of every product of every matrix appears exactly once (all
    256 x 256 tiles of B' X, the upper triangle for the symmetric A and B');
  * an item waits exactly for the previous stage of its own matrix, complete;
  * the table is topologically ordered: when an item is claimed, every item
    it waits for was claimed before it.  Claims happen only in running CTAs,
    so this order is what makes the schedule deadlock-free;
  * the table of k iterations is the prefix of the table of any larger k (the
    library builds the table once for 64 iterations and launches k of them).
"""
import numpy as np
import pytest

from paper_2608_05088_gb300 import build, inputs

SIGNALS_PER_ITEM = 16   # epilogue warps of a CTA pair


@pytest.fixture(scope="module")
def malt():
    build.build()
    import paper_2608_05088_gb300.malt as m
    return m


def cdiv(a, b):
    return (a + b - 1) // b


def expected_items(rows, cols, kind):
    p, q = min(rows, cols), max(rows, cols)
    tp, tq = cdiv(p, 256), cdiv(q, 256)
    if kind == 2:
        return tp * tq
    assert kind in (0, 1)
    return tp * (tp + 1) // 2


def check_table(tab, shapes, k):
    n = len(shapes)
    kinds = [0, 1, 2] * k
    seen = {}
    for grp, st, kind, mat, local, dep, target, nitems in tab:
        assert kind == kinds[st]
        rows, cols = shapes[mat]
        assert nitems == expected_items(rows, cols, kind), (st, kind, mat)
        seen.setdefault((int(st), int(mat)), []).append(int(local))
        if st == 0:
            assert dep == -1 and target == 0
        else:
            assert dep == (st - 1) * n + mat
            assert target == SIGNALS_PER_ITEM * expected_items(rows, cols, kinds[st - 1])
    assert set(seen) == {(s, i) for s in range(len(kinds)) for i in range(n)}
    for (st, mat), locs in seen.items():
        assert sorted(locs) == list(range(expected_items(*shapes[mat], kinds[st]))), (st, mat)
    # topological order per launch group: replay the claims with every item
    # finishing at once; each item's counter must be complete when claimed
    for grp in np.unique(tab[:, 0]):
        ctr = np.zeros(len(kinds) * n, dtype=np.int64)
        mats_here = set()
        for _, st, kind, mat, local, dep, target, nitems in tab[tab[:, 0] == grp]:
            mats_here.add(int(mat))
            if dep >= 0:
                assert ctr[dep] == target, (st, mat, local)
            ctr[st * n + mat] += SIGNALS_PER_ITEM
        # a matrix's whole step runs in one launch
        assert not mats_here & set(tab[tab[:, 0] != grp][:, 3].tolist())


RAGGED = [(200, 328), (392, 136), (8, 8), (136, 1000), (520, 520), (64, 2056), (1032, 264),
          (256, 512)]


@pytest.mark.parametrize("k", [1, 2, 5, 64])
def test_products_ragged(malt, k):
    check_table(malt.malt_ns_schedule(RAGGED, k), RAGGED, k)


def test_shorter_tables_are_prefixes(malt):
    """The library uploads one table for 64 iterations at init and launches
    the first k iterations' entries of it."""
    full = malt.malt_ns_schedule(RAGGED, 64)
    for k in (1, 3, 5, 17):
        tab = malt.malt_ns_schedule(RAGGED, k)
        for grp in np.unique(full[:, 0]):
            a, b = tab[tab[:, 0] == grp], full[full[:, 0] == grp]
            assert np.array_equal(a, b[: len(a)])
            assert len(b) == 64 * len(a) // k


def test_gpt2_large(malt):
    shapes = list(inputs.WORKLOADS["gpt2_large"].shapes)
    tab = malt.malt_ns_schedule(shapes, 5)
    check_table(tab, shapes, 5)
    # 36 of each of 1280x3840, 1280^2, 1280x5120, 5120x1280 (frames 1280 x
    # {3840, 1280, 5120, 5120}): 15 upper tiles per Gram / Poly, 5 x q/256 per BX
    per_iter = 144 * 15 * 2 + 36 * (5 * 15 + 5 * 5 + 2 * 5 * 20)
    assert len(tab) == 5 * per_iter
    # heaviest Gram reductions (q = 5120) are claimed first
    first = tab[: 72 * 15]
    assert all(max(shapes[m]) == 5120 for m in first[:, 3])


def test_more_classes_than_one_launch(malt):
    # ten distinct NS frames: two launch groups (at most eight classes each)
    shapes = [(64 * (i + 1), 512) for i in range(8)] + [(520, 8), (16, 16)]
    tab = malt.malt_ns_schedule(shapes, 3)
    assert set(np.unique(tab[:, 0]).tolist()) == {0, 1}
    check_table(tab, shapes, 3)


def test_unaligned_shapes_use_padded_frames(malt):
    """Rows and cols need not be multiples of 8: such a matrix runs on a
    zero-padded copy, so its table has the tiles of the padded frame, and a
    padded matrix shares a class with an aligned matrix of that frame."""
    odd = [(7, 13), (100, 3), (1001, 999), (250, 509), (256, 512), (1, 1)]
    padded = [(-(-m // 8) * 8, -(-n // 8) * 8) for m, n in odd]
    tab = malt.malt_ns_schedule(odd, 3)
    check_table(tab, padded, 3)


def test_bad_arguments(malt):
    with pytest.raises(malt.MaltError):
        malt.malt_ns_schedule([(256, 512)], 0)
    with pytest.raises(malt.MaltError):
        malt.malt_ns_schedule([(256, 512)], 65)
    with pytest.raises(malt.MaltError):
        malt.malt_ns_schedule([(0, 512)], 5)
