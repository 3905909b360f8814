"""Host-side logic of the BCD driver, on the CPU: the halo of an overlapping boundary region
and the culling rule for camera-partition pairs."""
import numpy as np

import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300.bcd import halo_members


def _cells(means, origin, side, dims):
    """Cell of each mean by brute force over every cell's closed box (lowest index on ties),
    clamped like the grid assignment for means outside the grid."""
    d = np.asarray(dims)
    ijk = np.clip(np.floor((means - origin) / side).astype(int), 0, d - 1)
    return ijk[:, 0] + d[0] * (ijk[:, 1] + d[1] * ijk[:, 2])


def test_halo_members_brute_force():
    rng = np.random.default_rng(3)
    dims, origin, side = (3, 2, 2), np.array([-7.5, -5.0, -5.0]), 5.0
    means = rng.uniform(origin, origin + side * np.array(dims), size=(3000, 3))
    cells = _cells(means, origin, side, dims)
    members = [np.nonzero(cells == c)[0] for c in range(12)]
    blocks = [c for c in range(12) if len(members[c])]
    for margin in (0.0, 0.7, 2.0):
        for b in (0, 4, 11):
            h = halo_members(means, members, blocks, b, dims, origin, side, margin)
            ix, iy, iz = b % 3, (b // 3) % 2, b // 6
            lo = origin + side * np.array([ix, iy, iz])
            hi = lo + side
            for q in blocks:
                if q == b:
                    assert q not in h
                    continue
                want = [k for k, i in enumerate(members[q])
                        if all(lo[a] - margin <= means[i, a] <= hi[a] + margin for a in range(3))]
                got = list(h.get(q, []))
                assert got == want, (margin, b, q)
            if margin == 0.0:                # only means exactly on b's faces (none here)
                assert not h
    # a margin as wide as the grid takes every other block whole
    h = halo_members(means, members, blocks, 4, dims, origin, side, 100.0)
    assert set(h) == set(blocks) - {4}
    assert all(len(h[q]) == len(members[q]) for q in h)


def test_cull_pairs_thresholds():
    v = np.array([0.2, 1e-4, 0.05, 0.0, 0.3])
    c = np.array([0.5, 0.4, 0.01, 0.0, 0.6])
    assert ab.cull_pairs(v, c, 0.0).tolist() == [True] * 5
    assert ab.cull_pairs(v, c, 1e-3).tolist() == [True, False, True, False, True]
    assert ab.cull_pairs(v, c, 1e-3, tau_area=0.02).tolist() == [True, False, False, False, True]
    assert ab.cull_pairs(v, c, 0.25).tolist() == [False, False, False, False, True]


def test_pair_visible_matches_oracle():
    """abcd_pair_visible (host code of libabcd) decides every pair as the oracle's restatement
    of the frustum rule does: walk-through and ring cameras, random boxes of every size."""
    import oracle
    from paper_2608_27735_gb300 import scenegen as sg
    ab.build()
    grid = sg.Grid(origin=np.array([-10.0, -10.0, -5.0]), side=5.0, dims=(4, 4, 2))
    cams = sg.inside_cameras(grid, 6, 160, 107, seed=3) + \
        sg.ring_cameras(6, 25.0, np.zeros(3), 160, 107, seed=3, height_jitter=1.0)
    rng = np.random.default_rng(12)
    agree = 0
    for cam in cams:
        c = ab.camera(cam)
        for _ in range(300):
            mid = rng.uniform(-20, 20, 3)
            h = rng.uniform(0.01, 6.0, 3)
            box = np.concatenate([mid - h, mid + h])
            assert ab.abcd_pair_visible(c, box) == oracle.pair_visible(cam, box), (mid, h)
            agree += 1
    assert agree == 12 * 300
