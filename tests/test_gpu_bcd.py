"""The block coordinate descent schedule over every block (Section 2) and the comparison of
Section 3 on a seeded synthetic scene: ABCD approaches full-scene training, the ablated
variant (blocks trained without F and B) does not."""
import numpy as np
import pytest

import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def test_abcd_matches_full_scene_quality_and_ablation_does_not():
    ab.build()
    from paper_2608_27735_gb300.bcd import quality_experiment
    h = quality_experiment(T=100, cycles=3)
    full, abcd, abl = h["full_scene"], h["abcd"], h["ablated"]
    assert full[-1] < 0.15 * full[0]
    assert abcd[-1] < 0.15 * abcd[0]
    assert abcd[-1] < 3.0 * full[-1]
    assert abl[-1] > 0.5 * abl[0] and abl[-1] > 5.0 * abcd[-1]
    # ABCD starts from the layered render of the same scene as the ablated variant
    assert abcd[0] == pytest.approx(abl[0], rel=1e-6)
    # culling the camera-partition pairs below a 1% visible share keeps ABCD's quality far
    # from the ablation's
    cul = h["abcd_culled"]
    assert cul[0] == pytest.approx(abcd[0], rel=1e-6)
    assert cul[-1] < 0.5 * abl[-1] and cul[-1] < 0.3 * cul[0]


def test_culling_at_zero_threshold_changes_nothing():
    """With a threshold of 0 every pair is kept: the stage composites the same layers in the
    same order and trains on the same cameras as without culling."""
    ab.build()
    from paper_2608_27735_gb300.bcd import BCD, default_lr
    s = sg.grid_scene((2, 1, 1), 5.0, 500, 0, seed=9)
    s.cameras = sg.ring_cameras(4, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 64, 48, seed=9)
    tg = np.stack([sg.random_image(48, 64, 3, seed=40 + k) for k in range(4)]).astype(np.float32)
    res = []
    for tau in (None, 0.0):
        run = BCD(s.gaussians, (2, 1, 1), s.grid.origin, 5.0, s.cameras, tg, 20, default_lr(10.0),
                  seed=4, cull_tau=tau)
        run.stage(run.blocks[0])
        res.append((run.loss.cpu().numpy(), run.F.cpu().numpy(), run.B.cpu().numpy(), run))
    np.testing.assert_allclose(res[0][0], res[1][0], rtol=1e-4)
    assert np.array_equal(res[0][1], res[1][1]) and np.array_equal(res[0][2], res[1][2])
    run = res[1][3]
    assert run.keep.all() and run.visible.shape == run.keep.shape
    # every camera's visible shares add up to the mean alpha of its full composite
    for ci in range(4):
        full = run.render_full(ci)[..., 3].double().mean().item()
        assert run.visible[ci].sum() == pytest.approx(full, abs=4 * 2.0 ** -23 + 1e-6)


def test_one_block_abcd_is_plain_training():
    """On a one-block grid F and B are transparent, so ABCD and its ablation run the same
    steps: the same losses up to the order of the backward's atomic sums."""
    ab.build()
    from paper_2608_27735_gb300.bcd import BCD, default_lr
    s = sg.grid_scene((1, 1, 1), 5.0, 600, 0, seed=7)
    s.cameras = sg.ring_cameras(4, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 64, 48, seed=7)
    tg = np.stack([sg.random_image(48, 64, 3, seed=20 + k) for k in range(4)]).astype(np.float32)
    res = []
    for mode in ("abcd", "ablated"):
        run = BCD(s.gaussians, (1, 1, 1), s.grid.origin, 5.0, s.cameras, tg, 40, default_lr(5.0),
                  mode=mode, seed=3)
        run.cycle()
        res.append((run.loss.cpu().numpy(), run.eval_loss()))
    np.testing.assert_allclose(res[0][0], res[1][0], rtol=1e-4)
    assert res[0][1] == pytest.approx(res[1][1], rel=1e-4)


def test_overlap_region_draws_every_gaussian_once():
    """The overlapping boundary region renders the neighbours' Gaussians near the block's faces
    with the block and leaves them out of F and B.  For the cameras on the split axis the
    layer order agrees with the depth order of every Gaussian, so the stage's composite, with
    or without the region, is the render of the whole scene with one depth sort, up to fp16 F
    and B and per-layer early termination (each Gaussian drawn exactly once); a region of
    width 0 is plain ABCD.  The cameras beside the split are where the layered composite
    departs from the one-sort render (reading R3); the gaps are returned for the record."""
    ab.build()
    from paper_2608_27735_gb300.bcd import BCD, default_lr
    s = sg.grid_scene((2, 1, 1), 5.0, 400, 0, seed=11)
    g = s.gaussians
    g.log_scales = (g.log_scales + np.log(4.0)).astype(np.float32)     # sigma ~ 1 of a cell of 5
    s.cameras = sg.ring_cameras(4, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 64, 48, seed=11)
    tg = np.zeros((4, 48, 64, 3), np.float32)
    lr = default_lr(10.0)
    full = BCD(g, (1, 1, 1), s.grid.origin, 10.0, s.cameras, tg, 0, lr)
    plain = BCD(g, (2, 1, 1), s.grid.origin, 5.0, s.cameras, tg, 0, lr)
    zero = BCD(g, (2, 1, 1), s.grid.origin, 5.0, s.cameras, tg, 0, lr, overlap=0.0)
    wide = BCD(g, (2, 1, 1), s.grid.origin, 5.0, s.cameras, tg, 0, lr, overlap=2.0)
    assert wide.halo[0] and wide.halo[1] and not zero.halo[0]
    side_gap = {"plain": 0.0, "wide": 0.0}
    for ci in range(4):                      # azimuths 0, 90, 180, 270 degrees
        ref = full.stage_render(full.blocks[0], ci)
        for b in (0, 1):
            p_, z_, w_ = plain.stage_render(b, ci), zero.stage_render(b, ci), wide.stage_render(b, ci)
            assert torch.equal(p_, z_)
            if ci in (0, 2):                 # on the split axis: exact up to fp16 and termination
                for o in (p_, w_):
                    d = (o - ref).abs()
                    assert d.mean().item() < 2e-3 and d.max().item() < 0.03, (ci, b, d.max().item())
            else:
                side_gap["plain"] += (p_ - ref).abs().mean().item()
                side_gap["wide"] += (w_ - ref).abs().mean().item()
    assert side_gap["plain"] > 1e-3              # beside the split the layering departs
    print("side-camera gap (mean |composite - one-sort render|, 4 renders):", side_gap)


def test_frustum_filter_of_camera_partition_pairs():
    """a0 (reading R14) with walk-through cameras inside a 4x4x2 grid: abcd_block_bounds holds
    the oracle's 3-sigma box of every block (to fp32 rounding), the driver's pair mask is the
    oracle's frustum rule on the cells united with those boxes, culled pairs are never cached,
    composited or trained on (their layers stay transparent), and a stage of a block trains on
    the cameras that see it only."""
    import oracle
    ab.build()
    from paper_2608_27735_gb300.bcd import BCD, default_lr
    s = sg.grid_scene((4, 4, 2), 5.0, 300, 0, seed=72)
    cams = sg.inside_cameras(s.grid, 8, 80, 54, seed=5)
    tg = np.stack([sg.random_image(54, 80, 3, seed=60 + k) for k in range(8)]).astype(np.float32)
    run = BCD(s.gaussians, s.grid.dims, s.grid.origin, s.grid.side, cams, tg, 6, default_lr(10.0),
              seed=2)
    cells = oracle.assign_cells(s.gaussians.means, s.grid.origin, s.grid.side, s.grid.dims)
    for b in run.blocks:
        gb = s.gaussians.subset(np.nonzero(cells == b)[0])
        ref = oracle.block_bounds(gb)
        box = torch.empty(6, device="cuda")
        ab.abcd_block_bounds(run.ctx, run.theta[b], box)
        run.ctx.sync()
        got = box.cpu().numpy().astype(np.float64)
        slack = 1e-5 * (1.0 + np.abs(ref))
        assert np.all(got[:3] <= ref[:3] + slack[:3]) and np.all(got[3:] >= ref[3:] - slack[3:])
        assert np.all(np.abs(got - ref) <= slack), (b, got, ref)
        ijk = np.array([b % 4, (b // 4) % 4, b // 16], np.float64)
        lo = np.asarray(s.grid.origin) + 5.0 * ijk
        full = np.concatenate([np.minimum(ref[:3], lo), np.maximum(ref[3:], lo + 5.0)])
        for ci, cam in enumerate(cams):
            assert run.frustum[ci, b] == oracle.pair_visible(cam, full), (ci, b)
    assert (~run.frustum).sum() >= 0.3 * run.frustum.size
    layers = run.layers.cpu()
    for ci in range(len(cams)):
        for b in run.blocks:
            if not run.frustum[ci, b]:
                assert int(layers[ci, b].abs().sum()) == 0
    b = max(run.blocks, key=lambda q: (0 < run.frustum[:, q].sum() < len(cams), run.frustum[:, q].sum()))
    allowed = set(run.cameras_of(b))
    assert allowed == {ci for ci in range(len(cams)) if run.frustum[ci, b]}
    seen = []
    run.stage(b, trace=lambda t, ci, *a: seen.append(ci))
    assert seen and set(seen) <= allowed
