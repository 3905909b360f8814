"""The other workload configurations at their own sizes, through the C ABI against the oracle:

* 3x3x3 grid x 20,000 Gaussians, SH degree 3, 640x480 (the centre partition, F and B from the
  26 others rendered by the oracle): every pixel and gradient, as for the tiny scene;
* the scene-scale workload the bench times (the active cell of a 4x4x2 grid x 100,000
  Gaussians, SH degree 3, 1237x822): sampled tiles' lists, every pixel of those tiles, and the
  gradient of every Gaussian for an upstream gradient on those tiles' unambiguous pixels;
* the cache compositing sweep at 1920x1080 with 64 layers: sampled pixels of F and B at
  several splits;
* the stress block (2,000,000 Gaussians from a 16-blob mixture, 1920x1080): as the
  scene-scale case.
Sampling keeps the oracle's share to seconds; the tiles are drawn with a fixed seed."""
import numpy as np
import pytest

import oracle
import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg
from tests import _parity as par
from tests.test_gpu_parity import Case, check_backward, run_forward

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def ctx():
    ab.build()
    c = ab.Context(0)
    c.reserve(200_000, 8_000_000, 2_100_000)
    return c


def test_config_medium_centre_partition(ctx):
    s = sg.medium_scene(n_cams=2)
    centre = 1 + 3 * (1 + 3 * 1)
    case = Case(s, 1, active=centre, fb=True)
    r = run_forward(ctx, case)
    R = oracle.render(case.sp, case.off, case.ids, case.cam.width, case.cam.height,
                      F=case.F64(), B=case.B64())
    n_alt = par.compare_render(r["out"].cpu().numpy(), r["state"].A_T.cpu().numpy()[..., 3], R,
                               case.sp, case.off, case.ids, case.P, case.opt, case.cam,
                               F=case.F64(), B=case.B64())
    # pixels resolved through the alternatives of a decision within rounding of its threshold
    assert n_alt < 0.05 * case.cam.width * case.cam.height
    check_backward(ctx, case, r, None, 21)


def sampled_block_check(ctx, g, cam_np, n_tiles_sampled, seed, max_pairs, min_clear=0.9):
    """Tile lists of sampled tiles, all pixels of those tiles, and grad2d of every Gaussian
    for an upstream gradient on those tiles' unambiguous pixels (zero elsewhere).  The oracle
    runs on the Gaussians that can reach the sampled tiles (under any admissible rounding):
    its lists of those tiles, and every pixel of them, are those of the whole block."""
    W, H = cam_np.width, cam_np.height
    tx, ty = oracle.tiles_xy(W, H)
    rng = np.random.default_rng(seed)
    tiles = np.sort(rng.choice(tx * ty, n_tiles_sampled, replace=False))
    P_all = oracle.project(g, cam_np)
    m_all, _ = par.margins(g, cam_np, P_all)
    sub = par.near_tiles(P_all, cam_np, m_all, tiles)
    gs = g.subset(sub)
    P = oracle.project(gs, cam_np)
    off, ids = oracle.tile_lists(P, W, H)
    m_uv, _ = par.margins(gs, cam_np, P)
    lo, hi, _ = par.rect_bounds(P, cam_np, m_uv)
    opt_list, opt = par.listing_ambiguity(P, lo, hi, cam_np, tiles=tiles, m_uv=m_uv)
    Fh, Bh = sg.premultiplied_layers(2, H, W, seed=seed + 1).astype(np.float16)
    F64, B64 = Fh.astype(np.float64), Bh.astype(np.float64)
    # GPU: the whole block
    cam = ab.camera(cam_np)
    theta = ab.Gaussians.from_numpy(g)
    proj = ab.Projected.alloc(theta.n)
    tl = ab.Tiles.alloc(max_pairs, W, H)
    ab.abcd_project(ctx, theta, cam, None, proj)
    ab.abcd_bin_sort(ctx, proj, theta.n, cam, tl)
    out = torch.empty(H, W, 4, device="cuda")
    st = ab.FwdState.alloc(W, H)
    Ft, Bt = torch.from_numpy(Fh).cuda(), torch.from_numpy(Bh).cuda()
    ab.abcd_render_composite_fwd(ctx, cam, None, proj, tl, Ft, Bt, ab.ABCD_F16, None, out, st)
    ctx.sync()
    K = int(tl.count.item())
    rng_gpu = tl.ranges.cpu().numpy().reshape(-1, 2).astype(np.int64)
    # GPU ids -> positions in the oracle's subset (ids outside it are in no sampled tile)
    pos = np.full(g.n, -1, np.int64)
    pos[sub] = np.arange(sub.size)
    gids = pos[tl.ids[:K].cpu().numpy().astype(np.int64)]
    par.check_tile_lists(rng_gpu, gids, off, ids, P, opt_list, tx * ty, tiles=tiles)
    # pixels of the sampled tiles
    sp = par.splats_with_margins(gs, cam_np, P)
    R = oracle.render(sp, off, ids, W, H, F=F64, B=B64)
    inside = np.zeros((H, W), bool)
    for t in tiles:
        y0, x0 = (t // tx) * 16, (t % tx) * 16
        inside[y0:y0 + 16, x0:x0 + 16] = True
    flagged = (R["n_ev"] > 0) | par.opt_pixel_mask(P, opt, cam_np)
    ok = inside & ~flagged
    # pixels with a decision within rounding of its threshold are left out; min_clear bounds
    # how many may be (deep, dense lists have many near the termination threshold)
    assert ok.sum() > min_clear * inside.sum()
    got = out.cpu().numpy()
    assert np.abs(got[ok] - R["out"][ok]).max() <= par.TOL_PIX
    assert np.abs(st.A_T.cpu().numpy()[..., 3][ok] - R["T_final"][ok]).max() <= par.TOL_PIX
    # gradients for an upstream gradient on the unambiguous sampled pixels
    G = np.zeros((H, W, 3))
    G[ok] = rng.normal(size=(int(ok.sum()), 3)) / (3.0 * H * W)
    G32 = G.astype(np.float32)
    grad2d = torch.empty(theta.n, 9, device="cuda")
    ab.abcd_render_backward(ctx, cam, None, proj, tl, Ft, Bt, ab.ABCD_F16, None, st,
                            torch.from_numpy(G32).cuda(), theta.n, grad2d)
    ctx.sync()
    ref_sub = oracle.backward_pixels(sp, off, ids, W, H, G32.astype(np.float64),
                                     np.flatnonzero(ok), F=F64, B=B64)
    ref = np.zeros((g.n, 9))
    ref[sub] = ref_sub
    assert np.abs(ref).max() > 0
    scale = np.abs(ref).max(0, keepdims=True)
    par.assert_grad_close(grad2d.cpu().numpy(), ref, rtol=1e-3, atol=1e-5 * scale, what="grad2d")
    return K


def test_config_scene_scale_sampled(ctx):
    s = sg.scene_scale(n_cams=3)
    cells = oracle.assign_cells(s.gaussians.means, s.grid.origin, s.grid.side, s.grid.dims)
    gx, gy, _ = s.grid.dims
    active = 1 + gx * (1 + gy * 0)                      # cell (1, 1, 0), as in the bench
    g = s.gaussians.subset(np.nonzero(cells == active)[0])
    assert g.n == 100_000
    ctx.reserve(g.n, 16_000_000, s.cameras[0].width * s.cameras[0].height)
    K = sampled_block_check(ctx, g, s.cameras[1], 160, seed=31, max_pairs=16_000_000)
    assert K > 1_000_000


def test_config_stress_block_sampled():
    g = sg.mixture_block(2_000_000, 10.0, 16, 3, seed=1004)
    cams = sg.ring_cameras(2, 12.0, np.zeros(3), 1920, 1080, seed=1004)
    c = ab.Context(0)                     # its own context: a capacity overflow is sticky
    cap = 400_000_000
    c.reserve(g.n, cap, 1920 * 1080)
    K = sampled_block_check(c, g, cams[0], 16, seed=41, max_pairs=cap, min_clear=0.3)
    assert K > 10_000_000


def test_config_cache_sweep_full_size_sampled(ctx):
    L, H, W = 64, 1080, 1920
    rng = np.random.default_rng(5)
    layers = sg.premultiplied_layers(L, H, W, seed=64).astype(np.float16)
    order = list(sg.random_permutation(L, seed=65))
    dev = [torch.from_numpy(layers[k]).cuda() for k in range(L)]
    pix = rng.choice(H * W, 4000, replace=False)
    sub = layers.reshape(L, H * W, 4)[:, pix].astype(np.float64)[:, :, None, :]   # [L][n][1][4]
    for split in (1, 31, 63):
        Fo = torch.empty(H, W, 4, dtype=torch.float16, device="cuda")
        Bo = torch.empty_like(Fo)
        lay = list(dev)
        lay[order[split]] = None
        ab.abcd_composite_cache(ctx, lay, order, split, W, H, Fo, Bo)
        ctx.sync()
        for got, ks in ((Fo, order[:split]), (Bo, order[split + 1:])):
            ref = oracle.composite_layers(sub, ks)[:, 0]
            g_ = got.reshape(H * W, 4)[torch.from_numpy(pix).cuda()].cpu().numpy()
            m = L * 4 * 2.0 ** -24 * np.abs(ref)
            lo_, hi_ = (ref - m).astype(np.float16), (ref + m).astype(np.float16)
            assert np.all((g_ >= lo_) & (g_ <= hi_)), split
            exact = lo_ == hi_
            assert np.all(g_[exact] == ref.astype(np.float16)[exact]), split
