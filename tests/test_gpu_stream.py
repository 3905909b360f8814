"""The out-of-core stage (paper_2608_27735_gb300/stream.py, Section 2's memory hierarchy) on the
GPU: K1 folded in pieces equals K1 at once bit for bit; a streamed stage equals the
device-resident stage; the peak device memory of a streamed stage is the same for a 2x2x2 and a
4x4x4 grid of 20,000-Gaussian partitions (O(1) in the scene's extent, Section 3); the disk tier
and checkpoint / resume give the same stages."""
import numpy as np
import pytest

import oracle
import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg
from paper_2608_27735_gb300.bcd import BCD, default_lr
from paper_2608_27735_gb300.stream import StreamingABCD

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def pack_layer(dense, tiles_x, tiles_y):
    """Test-side encoder of the packed layer format (a tile stored iff any of its pixels is not
    all-zero bits)."""
    H, W = dense.shape[:2]
    pad = np.zeros((tiles_y * 16, tiles_x * 16, 4), np.float16)
    pad[:H, :W] = dense
    blocks = pad.reshape(tiles_y, 16, tiles_x, 16, 4).transpose(0, 2, 1, 3, 4).reshape(-1, 16, 16, 4)
    used = np.any(blocks.view(np.uint16) != 0, axis=(1, 2, 3))
    tmap = np.where(used, np.cumsum(used) - 1, -1).astype(np.int32)
    return tmap, np.ascontiguousarray(blocks[used])


@pytest.fixture(scope="module")
def ctx():
    ab.build()
    c = ab.Context(0)
    c.reserve(1000, 1000, 200_000)
    return c


@pytest.mark.parametrize("H,W,L,piece", [(75, 101, 11, 3), (48, 64, 6, 1), (37, 29, 5, 4)])
def test_fold_in_pieces_equals_composite(ctx, H, W, L, piece):
    tx, ty = oracle.tiles_xy(W, H)
    st = sg.premultiplied_layers(L, H, W, seed=31 + L).astype(np.float16)
    rng = np.random.default_rng(L)
    for k in range(L):
        for t in np.nonzero(rng.random(tx * ty) < 0.4)[0]:
            y0, x0 = (t // tx) * 16, (t % tx) * 16
            st[k, y0:y0 + 16, x0:x0 + 16] = 0
    order = list(sg.random_permutation(L, seed=L))
    maps, packs = [], []
    for k in range(L):
        m, pk = pack_layer(st[k], tx, ty)
        maps.append(torch.from_numpy(m).cuda())
        packs.append(torch.from_numpy(pk if len(pk) else np.zeros((1, 16, 16, 4), np.float16)).cuda())
    for split in (0, L // 2, L):
        Fo = torch.empty(H, W, 4, dtype=torch.float16, device="cuda")
        Bo = torch.empty_like(Fo)
        Ff = torch.empty(H, W, 4, device="cuda")
        mm, pp = list(maps), list(packs)
        if split < L:
            mm[order[split]] = pp[order[split]] = None
        ab.abcd_composite_cache_packed(ctx, mm, pp, order, split, W, H, Fo, Bo)
        ab.abcd_composite_cache_packed(ctx, mm, pp, order, split, W, H, Ff, None, ab.ABCD_F32)
        for side, ref16 in ((order[:split], Fo), (order[split + 1:], Bo)):
            acc = torch.empty(H, W, 4, device="cuda")
            out16 = torch.full((H, W, 4), float("nan"), dtype=torch.float16, device="cuda")
            if not side:
                continue
            for j in range(0, len(side), piece):
                ks = side[j:j + piece]
                last = j + piece >= len(side)
                ab.abcd_composite_fold_packed(ctx, [maps[k] for k in ks], [packs[k] for k in ks], W, H,
                                              acc_in=acc if j else None, acc_out=acc,
                                              out16=out16 if last else None)
            ctx.sync()
            assert torch.equal(out16.view(torch.int16), ref16.view(torch.int16)), split
            if ref16 is Fo:
                assert torch.equal(acc, Ff), split


def _tiny_targets(scene, side):
    tgt = sg.perturbed(scene.gaussians, side, seed=2002)
    out = []
    for cam in scene.cameras:
        Pt = oracle.project(tgt, cam)
        ot, it = oracle.tile_lists(Pt, cam.width, cam.height)
        out.append(oracle.render(oracle.SplatSet.from_proj(Pt), ot, it, cam.width,
                                 cam.height)["out"][..., :3])
    return np.stack(out).astype(np.float32)


def test_streamed_stage_equals_resident_stage(tmp_path):
    """The same stage through host-resident layers (and through the disk tier) and through the
    device-resident driver: identical F and B, the same first loss bit for bit, the other losses
    and the parameters up to the order of the backward's atomic sums, and the refreshed layers."""
    scene = sg.tiny_scene(per_cell=800, res=96, n_cams=4)
    side, dims, origin = scene.grid.side, scene.grid.dims, scene.grid.origin
    targets = _tiny_targets(scene, side)
    lr = default_lr(2 * side)
    T = 8
    res = BCD(scene.gaussians, dims, origin, side, scene.cameras, targets, T, lr, seed=3)
    runs = [StreamingABCD(scene.gaussians, dims, origin, side, scene.cameras, targets, T, lr,
                          max_pairs=1_000_000, seed=3),
            StreamingABCD(scene.gaussians, dims, origin, side, scene.cameras, targets, T, lr,
                          max_pairs=1_000_000, seed=3, stage_tiles=40,
                          cache_dir=str(tmp_path / "disk"))]
    b = 3
    res.stage(b)
    res.ctx.sync()
    ref_loss = res.loss.cpu().numpy()
    for run in runs:
        loss = run.stage(b).numpy()
        assert loss[0] == ref_loss[0]
        np.testing.assert_allclose(loss, ref_loss, rtol=1e-4)
        for ci in range(len(scene.cameras)):
            assert torch.equal(run.host_F[ci].cuda().view(torch.int16), res.F[ci].view(torch.int16))
            assert torch.equal(run.host_B[ci].cuda().view(torch.int16), res.B[ci].view(torch.int16))
        for a_, t_ in zip(run.host_theta[b], res.theta[b].tensors()):
            np.testing.assert_allclose(a_.numpy(), t_.cpu().numpy(), rtol=1e-4, atol=1e-6)
        tx, ty = oracle.tiles_xy(96, 96)
        for ci in range(len(scene.cameras)):
            m, t = run.store.get(ci, b)
            dense = np.zeros((ty * 16, tx * 16, 4), np.float16)
            mm = m.numpy()
            for tile in range(tx * ty):
                if mm[tile] >= 0:
                    y0, x0 = (tile // tx) * 16, (tile % tx) * 16
                    dense[y0:y0 + 16, x0:x0 + 16] = t.numpy()[mm[tile]]
            ref = res.layers[ci, b].cpu().numpy().astype(np.float64)
            np.testing.assert_allclose(dense[:96, :96].astype(np.float64), ref, atol=2e-3)


def test_checkpoint_resume_gives_the_same_stage(tmp_path):
    scene = sg.tiny_scene(per_cell=500, res=64, n_cams=3)
    side, dims, origin = scene.grid.side, scene.grid.dims, scene.grid.origin
    targets = _tiny_targets(scene, side)
    lr = default_lr(2 * side)
    a = StreamingABCD(scene.gaussians, dims, origin, side, scene.cameras, targets, 4, lr,
                      max_pairs=500_000, seed=9)
    a.stage(0)
    a.save(str(tmp_path / "ckpt"))
    b = StreamingABCD(scene.gaussians, dims, origin, side, scene.cameras, targets, 4, lr,
                      max_pairs=500_000, seed=9)
    b.load(str(tmp_path / "ckpt"))
    b.rng, b.queue = np.random.default_rng(11), []
    a.rng, a.queue = np.random.default_rng(11), []
    for blk in a.blocks:
        for x, y in zip(a.host_theta[blk], b.host_theta[blk]):
            assert torch.equal(x, y)
    la, lb = a.stage(5).numpy(), b.stage(5).numpy()
    assert la[0] == lb[0]
    np.testing.assert_allclose(la, lb, rtol=1e-4)


def test_peak_device_memory_is_independent_of_scene_extent():
    """Section 3: for a fixed partition size and image resolution, the peak device memory of a
    stage does not depend on the number of partitions.  A 2x2x2 and a 4x4x4 grid of 20,000
    Gaussians per partition (SH 0, four 160x120 cameras): the same peak bytes allocated on the
    device over construction (initial cache of every block) and one stage; the host tier grows
    with the partitions."""
    peaks, host = {}, {}
    for dims in ((2, 2, 2), (4, 4, 4)):
        s = sg.grid_scene(dims, 5.0, 20_000, 0, seed=71)
        s.cameras = sg.ring_cameras(4, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 160, 120,
                                    seed=71, height_jitter=1.0)
        targets = np.zeros((4, 120, 160, 3), np.float32)
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        base = torch.cuda.memory_allocated()
        torch.cuda.reset_peak_memory_stats()
        run = StreamingABCD(s.gaussians, dims, s.grid.origin, 5.0, s.cameras, targets, 5,
                            default_lr(5.0), max_pairs=3_000_000, seed=1)
        run.stage(0)
        torch.cuda.synchronize()
        peaks[dims] = torch.cuda.max_memory_allocated() - base
        host[dims] = sum(t.numel() * t.element_size() for blk in run.host_theta.values() for t in blk)
        assert run.n_max == 20_000
        del run
    print(f"peak device bytes {peaks}; host parameter bytes {host}")
    assert peaks[(2, 2, 2)] == peaks[(4, 4, 4)]
    assert host[(4, 4, 4)] == 8 * host[(2, 2, 2)]
