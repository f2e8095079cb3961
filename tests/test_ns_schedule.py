"""The persistent Newton-Schulz schedule's work list, checked on the host.

The library computes the list with the same decode the kernel runs
(malt_ns_schedule needs no GPU).  The Orth step of Algorithm 1 iterates
A = X X^T, B' = aI + bA + cA^2, X <- B' X on each matrix's own data, so:
  * every 256 x 256 tile of every product of every iteration of every matrix
    appears exactly once (the upper triangle for the symmetric A and B');
  * a tile waits exactly for the previous product of its own matrix, complete;
  * the list is topologically ordered: when a tile is claimed, every tile it
    waits for was claimed before it.  Claims happen only in running CTAs, so
    this order is what makes the schedule deadlock-free.
"""
import numpy as np
import pytest

from paper_2608_05088_gb300 import build, inputs

SIGNALS_PER_TILE = 16   # epilogue warps of a CTA pair


@pytest.fixture(scope="module")
def malt():
    build.build()
    import paper_2608_05088_gb300.malt as m
    return m


def tiles(n):
    return (n + 255) // 256


def expected_tiles(rows, cols, s):
    p, q = min(rows, cols), max(rows, cols)
    kind = s % 3
    if kind == 2:
        return {(i, j) for i in range(tiles(p)) for j in range(tiles(q))}
    return {(i, j) for i in range(tiles(p)) for j in range(i, tiles(p))}


def check_schedule(sched, shapes, k):
    n = len(shapes)
    seen = {}
    for g, s, mat, mt, nt, dep, target, ntiles in sched:
        key = (int(s), int(mat))
        seen.setdefault(key, []).append((int(mt), int(nt)))
        rows, cols = shapes[mat]
        assert ntiles == len(expected_tiles(rows, cols, s))
        if s == 0:
            assert dep == -1
        else:
            assert dep == (s - 1) * n + mat
            assert target == SIGNALS_PER_TILE * len(expected_tiles(rows, cols, s - 1))
    assert set(seen) == {(s, i) for s in range(3 * k) for i in range(n)}
    for (s, mat), tl in seen.items():
        assert len(tl) == len(set(tl)), (s, mat)
        assert set(tl) == expected_tiles(*shapes[mat], s), (s, mat)
    # topological order per launch group: replay the claims with every tile
    # finishing at once; each tile's counter must be complete when claimed
    for grp in np.unique(sched[:, 0]):
        ctr = np.zeros(3 * k * n, dtype=np.int64)
        mats_here = set()
        for _, s, mat, mt, nt, dep, target, ntiles in sched[sched[:, 0] == grp]:
            mats_here.add(int(mat))
            if dep >= 0:
                assert ctr[dep] == target, (s, mat, mt, nt)
            ctr[s * n + mat] += SIGNALS_PER_TILE
        # a matrix's whole solve runs in one launch
        assert not mats_here & set(sched[sched[:, 0] != grp][:, 2].tolist())


RAGGED = [(200, 328), (392, 136), (8, 8), (136, 1000), (520, 520), (64, 2056), (1032, 264),
          (256, 512)]


@pytest.mark.parametrize("k", [1, 2, 5])
def test_ragged_shapes(malt, k):
    sched = malt.malt_ns_schedule(RAGGED, k)
    check_schedule(sched, RAGGED, k)


def test_gpt2_large(malt):
    shapes = list(inputs.WORKLOADS["gpt2_large"].shapes)
    sched = malt.malt_ns_schedule(shapes, 5)
    check_schedule(sched, shapes, 5)
    # 36 of each of 1280x3840, 1280^2, 1280x5120, 5120x1280 (frames 1280 x
    # {3840, 1280, 5120, 5120}): 15 upper tiles per Gram / Poly, 5 x q/256 per BX
    per_iter = 144 * 15 * 2 + 36 * (5 * 15 + 5 * 5 + 2 * 5 * 20)
    assert len(sched) == 5 * per_iter
    # heaviest Gram reductions (q = 5120) are claimed first
    first = sched[: 72 * 15]
    assert all(max(shapes[m]) == 5120 for m in first[:, 2])


def test_more_classes_than_one_launch(malt):
    # ten distinct NS frames: two launch groups (at most eight classes each)
    shapes = [(64 * (i + 1), 512) for i in range(8)] + [(520, 8), (16, 16)]
    sched = malt.malt_ns_schedule(shapes, 3)
    assert set(np.unique(sched[:, 0]).tolist()) == {0, 1}
    check_schedule(sched, shapes, 3)


def test_bad_arguments(malt):
    with pytest.raises(malt.MaltError):
        malt.malt_ns_schedule([(256, 512)], 0)
    with pytest.raises(malt.MaltError):
        malt.malt_ns_schedule([(256, 512)], 65)
    with pytest.raises(malt.MaltError):
        malt.malt_ns_schedule([(250, 512)], 5)
