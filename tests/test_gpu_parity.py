"""CUDA path (libabcd.so through its C ABI) versus the fp64 oracle on seeded inputs.

Tolerances: tile lists and sort order bit-exact (up to decisions the oracle proves are within
fp32 rounding of their threshold, see tests/_parity.py); pixels 1e-4 absolute; gradients 1e-3
relative or 1e-5 absolute; loss 1e-5 relative; fp16 outputs bit-exact except where the exact
value lies within fp32 accumulation error of an fp16 rounding midpoint.
"""
import math

import numpy as np
import pytest

import oracle
import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg
from tests import _parity as par

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def ctx():
    ab.build()
    c = ab.Context(0)
    c.reserve(200_000, 8_000_000, 2_100_000)
    return c


GROUPS = ("means", "log_scales", "quats", "opacity_logits", "sh")


class Case:
    """One seeded workload: the active block, a camera, F/B from the frozen partitions."""

    def __init__(self, scene, cam_idx, active=0, fb=True, fb_dtype="f16"):
        self.scene = scene
        self.cam = scene.cameras[cam_idx]
        g = scene.gaussians
        cells = oracle.assign_cells(g.means, scene.grid.origin, scene.grid.side, scene.grid.dims)
        self.g = g.subset(np.nonzero(cells == active)[0])
        self.F = self.B = None
        if fb:
            front, back = oracle.partition_split(scene.grid.dims, scene.grid.origin,
                                                 scene.grid.side, self.cam.position, active)
            layers = {}
            for p in list(front) + list(back):
                gp = g.subset(np.nonzero(cells == p)[0])
                P = oracle.project(gp, self.cam)
                off, ids = oracle.tile_lists(P, self.cam.width, self.cam.height)
                layers[p] = oracle.render(oracle.SplatSet.from_proj(P), off, ids,
                                          self.cam.width, self.cam.height)["out"]
            H, W = self.cam.height, self.cam.width
            keys = sorted(layers)
            st = np.stack([layers[k] for k in keys]) if keys else np.zeros((0, H, W, 4))
            idx = {k: i for i, k in enumerate(keys)}
            F64 = oracle.composite_layers(st, [idx[k] for k in front]) if len(front) else np.zeros((H, W, 4))
            B64 = oracle.composite_layers(st, [idx[k] for k in back]) if len(back) else np.zeros((H, W, 4))
            dt = np.float16 if fb_dtype == "f16" else np.float32
            self.F = F64.astype(dt)
            self.B = B64.astype(dt)
        self.P = oracle.project(self.g, self.cam)
        self.off, self.ids = oracle.tile_lists(self.P, self.cam.width, self.cam.height)
        self.m_uv, _ = par.margins(self.g, self.cam, self.P)
        self.lo, self.hi, self.amb_r = par.rect_bounds(self.P, self.cam, self.m_uv)
        self.opt_list, self.opt = par.listing_ambiguity(self.P, self.lo, self.hi, self.cam,
                                                             m_uv=self.m_uv)
        self.sp = par.splats_with_margins(self.g, self.cam, self.P)

    def F64(self):
        return None if self.F is None else self.F.astype(np.float64)

    def B64(self):
        return None if self.B is None else self.B.astype(np.float64)


def run_forward(ctx, case, bg=None, opts=None, want_state=True, refresh=False):
    cam = ab.camera(case.cam)
    theta = ab.Gaussians.from_numpy(case.g)
    proj = ab.Projected.alloc(theta.n)
    ab.abcd_project(ctx, theta, cam, opts, proj)
    tiles = ab.Tiles.alloc(4_000_000, case.cam.width, case.cam.height)
    ab.abcd_bin_sort(ctx, proj, theta.n, cam, tiles, opts)
    H, W = case.cam.height, case.cam.width
    out = torch.empty(H, W, 4, device="cuda")
    st = ab.FwdState.alloc(W, H) if want_state else None
    Ft = None if case.F is None else torch.from_numpy(case.F).cuda()
    Bt = None if case.B is None else torch.from_numpy(case.B).cuda()
    fbd = ab.ABCD_F16 if (case.F is None or case.F.dtype == np.float16) else ab.ABCD_F32
    rf = torch.empty(H, W, 4, dtype=torch.float16, device="cuda") if refresh else None
    ab.abcd_render_composite_fwd(ctx, cam, opts, proj, tiles, Ft, Bt, fbd, bg, out, st, rf)
    ctx.sync()
    return dict(cam=cam, theta=theta, proj=proj, tiles=tiles, out=out, state=st, F=Ft, B=Bt,
                fbd=fbd, refresh=rf)


@pytest.fixture(scope="module")
def tiny():
    return sg.tiny_scene()


@pytest.fixture(scope="module")
def ragged():
    # ragged image (150x100: partial tiles on both axes), SH degree 3
    s = sg.grid_scene((2, 2, 1), 5.0, 1500, 3, seed=77)
    s.cameras = sg.ring_cameras(3, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 150, 100, seed=77,
                                height_jitter=1.0)
    return s


# ----------------------------------------------------------------------------------------

@pytest.mark.parametrize("cam_idx", [0, 1, 2, 3])
def test_project_matches_oracle(ctx, tiny, cam_idx):
    case = Case(tiny, cam_idx, fb=False)
    r = run_forward(ctx, case, want_state=False)
    pr = r["proj"]
    P = case.P
    depth = pr.depth.cpu().numpy()
    np.testing.assert_array_equal(depth.view(np.uint32)[P["depth"] > 0.2], P["depth_key"][P["depth"] > 0.2])
    rad = pr.radius.cpu().numpy()
    vis = P["visible"] == 1
    exact = ~case.amb_r & vis & np.all(case.lo == case.hi, axis=1)
    np.testing.assert_array_equal(rad[exact], P["radius"][exact])
    assert np.all((rad > 0) == vis) or np.all(((rad > 0) != vis) <= ~np.all(case.lo == case.hi, axis=1))
    uv = pr.uv.cpu().numpy()
    co = pr.conic_opacity.cpu().numpy()
    rgb = pr.rgb.cpu().numpy()
    both = vis & (rad > 0)
    np.testing.assert_allclose(uv[both], P["uv"][both], rtol=0, atol=1e-3)
    np.testing.assert_allclose(co[both, 3], P["opacity"][both], rtol=1e-6, atol=1e-7)
    np.testing.assert_allclose(rgb[both], P["rgb"][both], rtol=1e-5, atol=1e-6)
    # conic: relative to its own scale (|a| + |c|)
    scale = (np.abs(P["conic"][both, 0]) + np.abs(P["conic"][both, 2]))[:, None]
    assert np.all(np.abs(co[both, :3] - P["conic"][both]) <= 1e-4 * scale)
    tt = pr.tiles_touched.cpu().numpy()
    nom = (P["rect"][:, 2] - P["rect"][:, 0]) * (P["rect"][:, 3] - P["rect"][:, 1])
    np.testing.assert_array_equal(tt[exact], nom[exact])


@pytest.mark.parametrize("cam_idx", [0, 1, 2, 3])
def test_bin_sort_matches_oracle(ctx, tiny, cam_idx):
    case = Case(tiny, cam_idx, fb=False)
    r = run_forward(ctx, case, want_state=False)
    K = int(r["tiles"].count.item())
    rng = r["tiles"].ranges.cpu().numpy().astype(np.int64)
    ids = r["tiles"].ids.cpu().numpy()[:K]
    tx, ty = oracle.tiles_xy(case.cam.width, case.cam.height)
    par.check_tile_lists(rng, ids, case.off, case.ids, case.P, case.opt_list, tx * ty)
    n_opt, share = par.optional_share(case.opt_list, K)
    print(f"camera {cam_idx}: K = {K}, oracle {len(case.ids)}, optional entries {n_opt} "
          f"({share:.2e} of K)")
    assert abs(K - len(case.ids)) <= n_opt
    assert share <= 1e-3


def test_bin_sort_ragged_and_sh3(ctx, ragged):
    for ci in range(3):
        case = Case(ragged, ci, fb=False)
        r = run_forward(ctx, case, want_state=False)
        K = int(r["tiles"].count.item())
        rng = r["tiles"].ranges.cpu().numpy().astype(np.int64)
        ids = r["tiles"].ids.cpu().numpy()[:K]
        tx, ty = oracle.tiles_xy(case.cam.width, case.cam.height)
        par.check_tile_lists(rng, ids, case.off, case.ids, case.P, case.opt_list, tx * ty)


def test_bin_sort_many_gaussians(ctx):
    """270,000 Gaussians: the depth sort's one-sweep passes span 132 tiles (long look-back
    chains), and the tile sort sees ids of 19 bits."""
    s = sg.grid_scene((1, 1, 1), 5.0, 270_000, 0, seed=91)
    s.cameras = sg.ring_cameras(1, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 96, 64, seed=91,
                                height_jitter=1.0)
    ctx.reserve(270_000, 8_000_000, 2_100_000)
    case = Case(s, 0, fb=False)
    r = run_forward(ctx, case, want_state=False)
    K = int(r["tiles"].count.item())
    rng = r["tiles"].ranges.cpu().numpy().astype(np.int64)
    ids = r["tiles"].ids.cpu().numpy()[:K]
    tx, ty = oracle.tiles_xy(case.cam.width, case.cam.height)
    par.check_tile_lists(rng, ids, case.off, case.ids, case.P, case.opt_list, tx * ty)


def test_bin_sort_depth_key_range(ctx):
    """The depth sort ranks keys relative to the smallest visible one, and a pass whose digit
    counts put every item in one bin runs as a copy (on ring cameras the last pass does).  The
    lists equal the oracle's where the visible keys span more than 2^24 values (a camera inside
    the block, depths from the near plane on: all four passes rank, the culled keys kept above
    the visible ones) and where nothing is visible (a camera looking away: no pair listed)."""
    s = sg.grid_scene((1, 1, 1), 5.0, 3000, 0, seed=97)
    c = np.asarray(s.grid.origin, dtype=np.float64) + 2.5
    s.cameras = [sg.look_at(c, c + np.array([1.0, 0.2, 0.1]), 96, 64),
                 sg.look_at(c - np.array([10.0, 0.0, 0.0]), c - np.array([20.0, 0.0, 0.0]), 96, 64)]
    ctx.reserve(3000, 2_000_000, 96 * 64)
    for ci in range(2):
        case = Case(s, ci, fb=False)
        vis = np.asarray(case.P["radius"]) > 0
        if ci == 0:
            bits = np.asarray(case.P["depth"], dtype=np.float32)[vis].view(np.uint32).astype(np.int64)
            assert bits.max() - bits.min() >= (1 << 24) and not vis.all()
        else:
            assert not vis.any() and len(case.ids) == 0
        r = run_forward(ctx, case, want_state=False)
        K = int(r["tiles"].count.item())
        rng = r["tiles"].ranges.cpu().numpy().astype(np.int64)
        ids = r["tiles"].ids.cpu().numpy()[:K]
        tx, ty = oracle.tiles_xy(case.cam.width, case.cam.height)
        par.check_tile_lists(rng, ids, case.off, case.ids, case.P, case.opt_list, tx * ty)
        if ci == 1:
            assert K == 0 and not rng.any()
            assert torch.count_nonzero(r["out"]).item() == 0


@pytest.mark.parametrize("W,H", [(4096, 640), (4200, 96), (64, 4200)])
def test_bin_sort_wide_image(ctx, W, H):
    """Large tile grids with 3,000 Gaussians; the lists equal the oracle's.  4096x640: 256 tile
    columns, the most that bin through tile-row runs; 4200x96: 263 columns, binned through
    sorted (tile, Gaussian) pairs (11 tile bits: passes of 6 and 5 bits); 64x4200: 263 tile
    rows, the runs sorted by row in two passes (5 and 4 bits)."""
    s = sg.grid_scene((1, 1, 1), 5.0, 3000, 0, seed=95)
    s.cameras = sg.ring_cameras(1, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), W, H, seed=95,
                                height_jitter=1.0)
    ctx.reserve(3000, 2_000_000, W * H)
    case = Case(s, 0, fb=False)
    r = run_forward(ctx, case, want_state=False)
    K = int(r["tiles"].count.item())
    rng = r["tiles"].ranges.cpu().numpy().astype(np.int64)
    ids = r["tiles"].ids.cpu().numpy()[:K]
    tx, ty = oracle.tiles_xy(case.cam.width, case.cam.height)
    assert tx * ty == ((W + 15) // 16) * ((H + 15) // 16)
    par.check_tile_lists(rng, ids, case.off, case.ids, case.P, case.opt_list, tx * ty)
    n_opt, share = par.optional_share(case.opt_list, K)
    print(f"{W}x{H}: K = {K}, optional entries {n_opt} ({share:.2e} of K)")


@pytest.mark.parametrize("cam_idx,bg,fbdt", [(0, None, "f16"), (1, (0.2, 0.5, 0.9), "f16"),
                                             (2, None, "f32"), (3, (1.0, 1.0, 1.0), "f16")])
def test_render_composite_fwd_matches_oracle(ctx, tiny, cam_idx, bg, fbdt):
    case = Case(tiny, cam_idx, fb=True, fb_dtype=fbdt)
    r = run_forward(ctx, case, bg=bg)
    R = oracle.render(case.sp, case.off, case.ids, case.cam.width, case.cam.height,
                      F=case.F64(), B=case.B64(), bg=bg)
    gout = r["out"].cpu().numpy()
    gT = r["state"].A_T.cpu().numpy()[..., 3]
    n_alt = par.compare_render(gout, gT, R, case.sp, case.off, case.ids, case.P, case.opt,
                               case.cam, F=case.F64(), B=case.B64(), bg=bg)
    assert n_alt < 0.01 * case.cam.width * case.cam.height
    # the saved active layer A also matches (state used by the backward pass)
    A = r["state"].A_T.cpu().numpy()[..., :3]
    ok = (R["n_ev"] == 0) & ~par.opt_pixel_mask(case.P, case.opt, case.cam)
    tx, _ = oracle.tiles_xy(case.cam.width, case.cam.height)
    assert np.abs(A[ok] - R["A"][..., :3][ok]).max() <= 1e-4
    # list positions agree wherever the GPU list equals the oracle's
    nl = r["state"].n_last.cpu().numpy()
    rng = r["tiles"].ranges.cpu().numpy().astype(np.int64)
    gids = r["tiles"].ids.cpu().numpy()
    same = np.zeros_like(ok)
    for t in range(rng.shape[0]):
        if list(gids[rng[t, 0]:rng[t, 1]]) == list(case.ids[case.off[t]:case.off[t + 1]]):
            same[(t // tx) * 16:(t // tx) * 16 + 16, (t % tx) * 16:(t % tx) * 16 + 16] = True
    assert np.all(nl[ok & same] == R["n_used"][ok & same])


def test_render_ragged_no_fb(ctx, ragged):
    case = Case(ragged, 1, fb=False)
    r = run_forward(ctx, case)
    R = oracle.render(case.sp, case.off, case.ids, case.cam.width, case.cam.height)
    par.compare_render(r["out"].cpu().numpy(), r["state"].A_T.cpu().numpy()[..., 3], R, case.sp,
                       case.off, case.ids, case.P, case.opt, case.cam)


def test_refresh_fp16_matches_oracle(ctx, tiny):
    """Cache refresh (Section 2): the active layer alone, premultiplied, rounded to fp16."""
    case = Case(tiny, 0, fb=False)
    r = run_forward(ctx, case, refresh=True)
    R = oracle.render(case.sp, case.off, case.ids, case.cam.width, case.cam.height)
    got = r["refresh"].cpu().numpy()
    ref = R["A"]
    ok = (R["n_ev"] == 0) & ~par.opt_pixel_mask(case.P, case.opt, case.cam)
    # fp16 of the fp32 value: equal to the RNE rounding of the exact value unless the exact
    # value is within 1e-4 (the fp32 pixel tolerance) of an fp16 rounding midpoint
    lo = (ref - 1e-4).astype(np.float16)
    hi = (ref + 1e-4).astype(np.float16)
    g = got.astype(np.float64)
    assert np.all((g[ok] >= lo[ok].astype(np.float64)) & (g[ok] <= hi[ok].astype(np.float64)))
    exact = ok[..., None] & (lo == hi)
    assert np.all(got[exact] == ref.astype(np.float16)[exact])


def check_backward(ctx, case, r, bg, seed, state=None):
    """Render backward of a forward result `r` against the oracle's, for a seeded dL/dA."""
    H, W = case.cam.height, case.cam.width
    rng = np.random.default_rng(seed)
    G = (rng.normal(size=(H, W, 3)) / (3.0 * H * W)).astype(np.float32)
    grad2d = torch.empty(case.g.n, 9, device="cuda")
    ab.abcd_render_backward(ctx, r["cam"], None, r["proj"], r["tiles"], r["F"], r["B"], r["fbd"],
                            bg, state or r["state"], torch.from_numpy(G).cuda(), case.g.n, grad2d)
    ctx.sync()
    ref = oracle.backward(case.sp, case.off, case.ids, W, H, G.astype(np.float64), F=case.F64(),
                          B=case.B64(), bg=bg)
    R = oracle.render(case.sp, case.off, case.ids, W, H, F=case.F64(), B=case.B64(), bg=bg)
    lo, hi, npx = par.grad_envelope(case.sp, case.off, case.ids, case.P, case.opt, R, case.cam,
                                    G.astype(np.float64), F=case.F64(), B=case.B64(), bg=bg)
    # absolute floor: 1e-5 of each component's largest magnitude (G is scaled like a loss
    # gradient, so this is stricter than a fixed 1e-5)
    scale = np.abs(ref).max(0, keepdims=True)
    par.assert_grad_close(grad2d.cpu().numpy(), ref, lo, hi, rtol=1e-3, atol=1e-5 * scale,
                          what="grad2d")
    return R


@pytest.mark.parametrize("cam_idx", [0, 2])
def test_render_backward_matches_oracle(ctx, tiny, cam_idx):
    case = Case(tiny, cam_idx, fb=True)
    bg = (0.1, 0.2, 0.3)
    r = run_forward(ctx, case, bg=bg)
    check_backward(ctx, case, r, bg, 100 + cam_idx)


CK_CHUNK = 128   # list positions between the render checkpoints


def faint_scene(n, width, height, seed=93):
    """One cell of n faint Gaussians (opacity logits N(-5, 0.3^2)): tile lists of thousands of
    entries that the pixels stay open through, so the backward splits them into many chunks."""
    s = sg.grid_scene((1, 1, 1), 5.0, n, 0, seed=seed)
    s.cameras = sg.ring_cameras(1, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), width, height,
                                seed=seed, height_jitter=1.0)
    g = s.gaussians
    g.opacity_logits[:] = (-5.0 + 0.3 * np.random.default_rng(seed).normal(size=g.n)).astype(np.float32)
    return s


@pytest.fixture(scope="module")
def faint():
    return faint_scene(60_000, 64, 48)


def test_render_backward_long_walks(ctx, faint):
    """Walks of up to ~13,500 list positions: past the 32 chunks a block can list, so its last
    listed chunk runs to the end of the walk."""
    case = Case(faint, 0, fb=False)
    assert np.diff(case.off).max() > 33 * CK_CHUNK
    r = run_forward(ctx, case)
    R = oracle.render(case.sp, case.off, case.ids, case.cam.width, case.cam.height)
    par.compare_render(r["out"].cpu().numpy(), r["state"].A_T.cpu().numpy()[..., 3], R, case.sp,
                       case.off, case.ids, case.P, case.opt, case.cam)
    assert R["n_used"].max() > 33 * CK_CHUNK
    check_backward(ctx, case, r, None, 7)
    # a second backward of the same forward reuses its checkpoints
    check_backward(ctx, case, r, None, 8)


def test_render_backward_checkpoint_buffer_full():
    """A context sized for a 96x64 image holds 1,024 chunk checkpoints, fewer than the faint
    scene's long walks ask for: blocks that find the buffer full walk on to their end."""
    c = ab.Context(0)
    c.reserve(60_000, 1_000_000, 96 * 64)
    case = Case(faint_scene(60_000, 96, 64), 0, fb=False)
    r = run_forward(c, case)
    n_chunks = sum(max(0, (int(n) - 1) // CK_CHUNK) for n in np.diff(case.off)) * 4
    assert n_chunks > 1024
    check_backward(c, case, r, None, 9)


def test_render_backward_after_other_forward(ctx, tiny):
    """A forward into another state replaces the checkpoints; the backward of the first state
    then walks each block whole and still matches."""
    case = Case(tiny, 1, fb=True)
    bg = (0.3, 0.3, 0.3)
    r = run_forward(ctx, case, bg=bg)
    run_forward(ctx, Case(tiny, 3, fb=False))
    check_backward(ctx, case, r, bg, 11)


def test_project_backward_matches_oracle(ctx, ragged):
    case = Case(ragged, 0, fb=False)
    theta = ab.Gaussians.from_numpy(case.g)
    rng = np.random.default_rng(5)
    vis = case.P["visible"] == 1
    g2 = (rng.normal(size=(case.g.n, 9)) * vis[:, None]).astype(np.float32)
    g2[:, 2:5] *= 10.0
    grads = ab.Gaussians.zeros_like(theta)
    ab.abcd_project_backward(ctx, theta, ab.camera(case.cam), None, torch.from_numpy(g2).cuda(), grads)
    ctx.sync()
    ref = oracle.project_backward(case.g, case.cam, g2.astype(np.float64))
    clamp_near = np.any(np.abs(case.P["rgb_raw"]) < 1e-5, axis=1)
    keep = ~clamp_near
    for name, t in zip(("means", "log_scales", "quats", "opacity_logits", "sh"), grads.tensors()):
        got = t.cpu().numpy()[keep]
        r = ref[name][keep]
        s = np.abs(r).max()
        # absolute floor: 1e-5, or 1e-5 of the largest component when that is smaller
        par.assert_grad_close(got, r, rtol=1e-3, atol=min(1e-5, 1e-5 * s), what=name)


def test_loss_matches_oracle(ctx):
    # sizes below, at and across the 118x16 tiles of the two loss kernels (ragged tails in both
    # directions, several tiles in each) and of the fused kernel's 64x28 tiles
    for (H, W, lam, seed) in [(64, 64, 0.2, 1), (100, 150, 0.2, 2), (37, 53, 0.0, 3), (128, 96, 1.0, 4),
                              (70, 300, 0.2, 5), (9, 13, 0.2, 6), (33, 237, 0.5, 7)]:
        x = sg.random_image(H, W, 4, seed)
        y = np.clip(x[..., :3] + sg.random_image(H, W, 3, seed + 50, -0.2, 0.2), 0, 1).astype(np.float32)
        L, g = oracle.loss(x[..., :3].astype(np.float64), y.astype(np.float64), lam)
        lt = torch.zeros(1, device="cuda")
        gt = torch.empty(H, W, 3, device="cuda")
        ab.abcd_loss(ctx, torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda(), W, H, lam, lt, gt)
        ctx.sync()
        assert abs(lt.item() - L) <= 1e-5 * abs(L), (H, W, lam, lt.item(), L)
        got = gt.cpu().numpy().astype(np.float64)
        tol = 1e-3 * np.abs(g) + 1e-6 * np.abs(g).max()
        assert np.all(np.abs(got - g) <= tol), (H, W, lam, np.abs(got - g).max())


@pytest.mark.parametrize("dtype,out_dtype,H,W,L", [("f16", "f16", 48, 64, 9), ("f16", "f16", 37, 29, 5),
                                                    ("f32", "f32", 40, 40, 7), ("f16", "f32", 17, 33, 12)])
def test_composite_cache_matches_oracle(ctx, dtype, out_dtype, H, W, L):
    st = sg.premultiplied_layers(L, H, W, seed=L)
    order = list(sg.random_permutation(L, seed=H))
    ldt = np.float16 if dtype == "f16" else np.float32
    layers_np = st.astype(ldt)
    layers = [torch.from_numpy(layers_np[k]).cuda() for k in range(L)]
    for split in (0, L // 2, L - 1, L):
        odt = torch.float16 if out_dtype == "f16" else torch.float32
        Fo = torch.empty(H, W, 4, dtype=odt, device="cuda")
        Bo = torch.empty(H, W, 4, dtype=odt, device="cuda")
        lay = list(layers)
        if split < L:
            lay[order[split]] = None        # the active partition's own layer is skipped
        ab.abcd_composite_cache(ctx, lay, order, split, W, H, Fo, Bo,
                                ab.ABCD_F16 if dtype == "f16" else ab.ABCD_F32,
                                ab.ABCD_F16 if out_dtype == "f16" else ab.ABCD_F32)
        ctx.sync()
        src = layers_np.astype(np.float64)
        Fr = oracle.composite_layers(src, order[:split]) if split > 0 else np.zeros((H, W, 4))
        Br = oracle.composite_layers(src, order[split + 1:]) if split + 1 < L else np.zeros((H, W, 4))
        for got, ref in ((Fo, Fr), (Bo, Br)):
            g = got.cpu().numpy()
            if out_dtype == "f32":
                assert np.abs(g - ref).max() <= 1e-6
            else:
                # fp32 accumulation of non-negative terms: every partial sum is <= the result,
                # so the accumulated rounding is <= L * 4 u * result
                m = L * 4 * 2.0 ** -24 * np.abs(ref)
                lo, hi = (ref - m).astype(np.float16), (ref + m).astype(np.float16)
                assert np.all((g >= lo) & (g <= hi))
                exact = lo == hi
                assert np.all(g[exact] == ref.astype(np.float16)[exact])
                assert exact.mean() > 0.99


def check_fb16(got, ref, L):
    """fp16 composite output against the exact fold (fp32 accumulation, one rounding)."""
    g = got.cpu().numpy()
    m = L * 4 * 2.0 ** -24 * np.abs(ref)
    lo, hi = (ref - m).astype(np.float16), (ref + m).astype(np.float16)
    assert np.all((g >= lo) & (g <= hi))
    exact = lo == hi
    assert np.all(g[exact] == ref.astype(np.float16)[exact])


def test_cache_host_tier_streams_layers(ctx):
    """Host tier of the cache: two cameras' layers come from pinned host memory through ONE
    device buffer (fetch on the copy stream, wait, composite, release), so the second fetch
    must not land before the first composite has read the buffer; a composite goes back to
    the host with a store."""
    L, H, W = 6, 70, 90
    cams = [sg.premultiplied_layers(L, H, W, seed=300 + c).astype(np.float16) for c in range(2)]
    host = [torch.from_numpy(x).pin_memory() for x in cams]
    dev = torch.empty(L, H, W, 4, dtype=torch.float16, device="cuda")
    order = list(sg.random_permutation(L, seed=31))
    split = 2
    outs = []
    for c in range(2):
        ab.abcd_cache_fetch(ctx, 0, host[c], dev)
        ab.abcd_cache_wait(ctx, 0)
        Fo = torch.empty(H, W, 4, dtype=torch.float16, device="cuda")
        Bo = torch.empty_like(Fo)
        lay = [dev[k] for k in range(L)]
        lay[order[split]] = None
        ab.abcd_composite_cache(ctx, lay, order, split, W, H, Fo, Bo)
        ab.abcd_cache_release(ctx, 0)
        outs.append((Fo, Bo))
    back = torch.empty(H, W, 4, dtype=torch.float16).pin_memory()
    ab.abcd_cache_store(ctx, 1, outs[1][0], back)
    ctx.sync()
    ab.abcd_cache_sync(ctx)
    for c in range(2):
        src = cams[c].astype(np.float64)
        check_fb16(outs[c][0], oracle.composite_layers(src, order[:split]), L)
        check_fb16(outs[c][1], oracle.composite_layers(src, order[split + 1:]), L)
    assert torch.equal(back, outs[1][0].cpu())
    with pytest.raises(ab.AbcdError):
        ab.abcd_cache_fetch(ctx, ab.ABCD_MAX_CACHE_SLOTS, host[0], dev)
    with pytest.raises(ab.AbcdError):
        ab.abcd_cache_wait(ctx, -1)


def pack_layer(dense, tiles_x, tiles_y):
    """Test-side encoder of the packed layer format: (tile_map, packed) of a dense fp16
    [H][W][4] layer, a tile stored iff any of its pixels is not all-zero bits."""
    H, W = dense.shape[:2]
    pad = np.zeros((tiles_y * 16, tiles_x * 16, 4), np.float16)
    pad[:H, :W] = dense
    blocks = pad.reshape(tiles_y, 16, tiles_x, 16, 4).transpose(0, 2, 1, 3, 4).reshape(-1, 16, 16, 4)
    used = np.any(blocks.view(np.uint16) != 0, axis=(1, 2, 3))
    tmap = np.where(used, np.cumsum(used) - 1, -1).astype(np.int32)
    return tmap, np.ascontiguousarray(blocks[used])


def test_refresh_packed_matches_dense_refresh(ctx, ragged):
    """K10 into the packed format: the stored tiles are the dense refresh's, bit for bit, and
    every tile left out is transparent in it."""
    case = Case(ragged, 2, fb=False)
    r = run_forward(ctx, case, want_state=False, refresh=True)
    W, H = case.cam.width, case.cam.height
    tx, ty = oracle.tiles_xy(W, H)
    tmap = torch.full((tx * ty,), -7, dtype=torch.int32, device="cuda")
    packed = torch.zeros(tx * ty, 16, 16, 4, dtype=torch.float16, device="cuda")
    count = torch.zeros(1, dtype=torch.int32, device="cuda")
    ab.abcd_render_refresh_packed(ctx, r["cam"], None, r["proj"], r["tiles"], tmap, packed, count)
    # the one-call form (project, bin_sort, packed refresh) gives the same bytes
    tmap2, packed2, count2 = torch.full_like(tmap, -7), torch.zeros_like(packed), torch.zeros_like(count)
    ab.RefreshLayer(ctx, r["theta"], ab.Projected.alloc(r["theta"].n),
                    ab.Tiles.alloc(4_000_000, W, H))(r["cam"], tmap2, packed2, count2)
    ctx.sync()
    assert torch.equal(tmap, tmap2) and torch.equal(count, count2)
    used2 = (tmap2 >= 0).nonzero().numel()
    assert torch.equal(packed2[:used2].view(torch.int16), packed[:used2].view(torch.int16))
    dense = r["refresh"].cpu().numpy()
    m = tmap.cpu().numpy()
    rng = r["tiles"].ranges.cpu().numpy().reshape(-1, 2).astype(np.int64)
    used = rng[:, 1] > rng[:, 0]
    assert np.array_equal(m >= 0, used) and int(count.item()) == int(used.sum())
    assert np.array_equal(m[used], np.arange(used.sum()))
    pk = packed.cpu().numpy()
    pad = np.zeros((ty * 16, tx * 16, 4), np.float16)
    pad[:H, :W] = dense
    blocks = pad.reshape(ty, 16, tx, 16, 4).transpose(0, 2, 1, 3, 4).reshape(-1, 16, 16, 4)
    inside = np.zeros((ty * 16, tx * 16), bool)
    inside[:H, :W] = True
    inb = inside.reshape(ty, 16, tx, 16).transpose(0, 2, 1, 3).reshape(-1, 16, 16)
    for t in range(tx * ty):
        if used[t]:
            ok = inb[t]
            assert np.array_equal(pk[m[t]][ok].view(np.uint16), blocks[t][ok].view(np.uint16)), t
        else:
            assert not np.any(blocks[t].view(np.uint16)), t


def test_composite_packed_matches_dense(ctx):
    """K1 over packed layers equals K1 over the dense layers bit for bit (a tile a layer leaves
    out folds like its zeros), on a ragged image with layers that leave tiles out."""
    L, H, W = 7, 75, 101
    tx, ty = oracle.tiles_xy(W, H)
    st = sg.premultiplied_layers(L, H, W, seed=17).astype(np.float16)
    rng = np.random.default_rng(5)
    for k in range(L):                      # blank a random third of each layer's tiles
        for t in np.nonzero(rng.random(tx * ty) < 0.33)[0]:
            y0, x0 = (t // tx) * 16, (t % tx) * 16
            st[k, y0:y0 + 16, x0:x0 + 16] = 0
    order = list(sg.random_permutation(L, seed=8))
    maps, packs = [], []
    for k in range(L):
        m, pk = pack_layer(st[k], tx, ty)
        maps.append(torch.from_numpy(m).cuda())
        packs.append(torch.from_numpy(pk if len(pk) else np.zeros((1, 16, 16, 4), np.float16)).cuda())
    dense = [torch.from_numpy(st[k]).cuda() for k in range(L)]
    for split in (0, 3, L):
        outs = []
        for packed_path in (False, True):
            Fo = torch.empty(H, W, 4, dtype=torch.float16, device="cuda")
            Bo = torch.empty_like(Fo)
            if packed_path:
                mm, pp = list(maps), list(packs)
                if split < L:
                    mm[order[split]] = pp[order[split]] = None
                ab.abcd_composite_cache_packed(ctx, mm, pp, order, split, W, H, Fo, Bo)
            else:
                lay = list(dense)
                if split < L:
                    lay[order[split]] = None
                ab.abcd_composite_cache(ctx, lay, order, split, W, H, Fo, Bo)
            outs.append((Fo, Bo))
        ctx.sync()
        for a_, b_ in zip(outs[0], outs[1]):
            assert torch.equal(a_.view(torch.int16), b_.view(torch.int16)), split


def _blank_tiles(st, tx, ty, share, seed):
    """Zero a random share of each layer's 16x16 tiles (the layers' transparent regions)."""
    rng = np.random.default_rng(seed)
    for k in range(st.shape[0]):
        for t in np.nonzero(rng.random(tx * ty) < share)[0]:
            y0, x0 = (t // tx) * 16, (t % tx) * 16
            st[k, y0:y0 + 16, x0:x0 + 16] = 0
    return st


def visibility_tol(count):
    """Mean of values rounded to 2^-24 fixed point (2^-25 each) after fp32 transmittance
    products of up to count factors (relative error <= count 2^-24)."""
    return 2.0 ** -24 + count * 2.0 ** -23


@pytest.mark.parametrize("H,W,L", [(37, 53, 9), (75, 101, 40), (16, 16, 1)])
def test_layer_visibility_matches_oracle(ctx, H, W, L):
    """Visible share and coverage of each layer of a depth order (dense and packed layers)
    against the oracle; the sums are exact integers, so packed equals dense bit for bit and a
    repeated call returns the same bits (the accumulators are cleared between calls)."""
    tx, ty = oracle.tiles_xy(W, H)
    st = _blank_tiles(sg.premultiplied_layers(L, H, W, seed=40 + L).astype(np.float16), tx, ty,
                      0.3, 6)
    src = st.astype(np.float64)
    dense = [torch.from_numpy(st[k]).cuda() for k in range(L)]
    maps, packs = [], []
    for k in range(L):
        m, pk = pack_layer(st[k], tx, ty)
        maps.append(torch.from_numpy(m).cuda())
        packs.append(torch.from_numpy(pk if len(pk) else np.zeros((1, 16, 16, 4), np.float16)).cuda())
    perm = list(sg.random_permutation(L, seed=H))
    for order in (perm, perm[: max(1, L // 2)], []):
        vr, cr = oracle.layer_visibility(src, order)
        got = []
        for packed_path in (False, True, True):
            vis = torch.full((L,), -1.0, dtype=torch.float64, device="cuda")
            cov = torch.full((L,), -1.0, dtype=torch.float64, device="cuda")
            if packed_path:
                ab.abcd_layer_visibility_packed(ctx, maps, packs, order, W, H, vis, cov)
            else:
                ab.abcd_layer_visibility(ctx, dense, order, W, H, vis, cov)
            ctx.sync()
            got.append((vis.cpu().numpy(), cov.cpu().numpy()))
        tol = visibility_tol(len(order))
        np.testing.assert_allclose(got[0][0], vr, rtol=0, atol=tol)
        np.testing.assert_allclose(got[0][1], cr, rtol=0, atol=tol)
        for g in got[1:]:
            assert np.array_equal(g[0], got[0][0]) and np.array_equal(g[1], got[0][1])


def test_layer_visibility_occlusion_and_errors(ctx):
    """An opaque layer in front hides every layer behind it exactly; coverage ignores it; a
    culled composite stays within the bound the dropped layers' visible shares give; bad
    orders are refused before any launch."""
    L, H, W = 5, 40, 50
    st = sg.premultiplied_layers(L, H, W, seed=77).astype(np.float16)
    st[2, :, :, :] = 0
    st[2, :, :, 3] = 1                       # an opaque black layer
    dense = [torch.from_numpy(st[k]).cuda() for k in range(L)]
    vis = torch.empty(L, dtype=torch.float64, device="cuda")
    cov = torch.empty(L, dtype=torch.float64, device="cuda")
    ab.abcd_layer_visibility(ctx, dense, [4, 2, 0, 1, 3], W, H, vis, cov)
    ctx.sync()
    v, c = vis.cpu().numpy(), cov.cpu().numpy()
    assert v[0] == 0 and v[1] == 0 and v[3] == 0 and v[2] > 0
    np.testing.assert_allclose(c, st[..., 3].astype(np.float64).mean(axis=(1, 2)), atol=visibility_tol(L))
    # culling by a threshold: the culled composite (abcd_composite_cache over the kept layers)
    # is within the dropped layers' visible shares of the full one, channel by channel
    st = sg.premultiplied_layers(L, H, W, seed=78).astype(np.float16)
    st[1] *= np.float16(0.01)
    st[3] *= np.float16(0.02)
    dense = [torch.from_numpy(st[k]).cuda() for k in range(L)]
    order = [0, 1, 2, 3, 4]
    ab.abcd_layer_visibility(ctx, dense, order, W, H, vis, cov)
    full = torch.empty(H, W, 4, device="cuda")
    ab.abcd_composite_cache(ctx, dense, order, L, W, H, full, None, ab.ABCD_F16, ab.ABCD_F32)
    ctx.sync()
    v, c = vis.cpu().numpy(), cov.cpu().numpy()
    keep = ab.cull_pairs(v, c, tau_visible=0.02)
    assert not keep[1] and not keep[3] and keep[[0, 2, 4]].all()
    kept = [j for j in order if keep[j]]
    culled = torch.empty(H, W, 4, device="cuda")
    ab.abcd_composite_cache(ctx, [dense[j] for j in kept], list(range(len(kept))), len(kept),
                            W, H, culled, None, ab.ABCD_F16, ab.ABCD_F32)
    ctx.sync()
    err = (full - culled).abs().double().mean(dim=(0, 1)).cpu().numpy()
    assert np.all(err <= v[~keep].sum() + 1e-6), (err, v[~keep])
    for bad in ([0, 0], [0, 5], [-1]):
        with pytest.raises(ab.AbcdError):
            ab.abcd_layer_visibility(ctx, dense, bad, W, H, vis, cov)


def test_adam_matches_oracle(ctx, ragged):
    g = ragged.gaussians.subset(slice(0, 3001))
    theta = ab.Gaussians.from_numpy(g)
    rng = np.random.default_rng(9)
    gr = [rng.normal(size=t.shape).astype(np.float32) for t in theta.tensors()]
    grads = ab.Gaussians(*(torch.from_numpy(a).cuda() for a in gr), g.sh_degree)
    m = ab.Gaussians.zeros_like(theta)
    v = ab.Gaussians.zeros_like(theta)
    lr = [1.6e-4, 5e-3, 1e-3, 0.025, 2.5e-3, 2.5e-3 / 20]
    ref = [a.astype(np.float64).copy() for a in g.arrays()]
    mr = [np.zeros_like(a) for a in ref]
    vr = [np.zeros_like(a) for a in ref]
    for step in (1, 2, 3):
        ab.abcd_adam_active(ctx, theta, grads, m, v, lr, 0.9, 0.999, 1e-15, step)
        for k in range(5):
            if k < 4:
                oracle.adam(ref[k], gr[k], mr[k], vr[k], lr[k], 0.9, 0.999, 1e-15, step)
            else:   # SH: degree-0 coefficients and the rest have their own learning rates
                for sl, l in ((np.s_[:, :1, :], lr[4]), (np.s_[:, 1:, :], lr[5])):
                    a, mm, vv = (np.ascontiguousarray(x[sl]) for x in (ref[4], mr[4], vr[4]))
                    oracle.adam(a, np.ascontiguousarray(gr[4][sl]), mm, vv, l, 0.9, 0.999, 1e-15, step)
                    ref[4][sl], mr[4][sl], vr[4][sl] = a, mm, vv
    ctx.sync()
    for k, t in enumerate(theta.tensors()):
        np.testing.assert_allclose(t.cpu().numpy(), ref[k], rtol=2e-6, atol=2e-7)


def _full_step(ctx, scene, case):
    H, W = case.cam.height, case.cam.width
    tgt = sg.perturbed(scene.gaussians, scene.grid.side, seed=2002)
    Pt = oracle.project(tgt, case.cam)
    ot, it = oracle.tile_lists(Pt, W, H)
    gt = oracle.render(oracle.SplatSet.from_proj(Pt), ot, it, W, H)["out"][..., :3].astype(np.float32)
    r = run_forward(ctx, case)
    loss = torch.zeros(1, device="cuda")
    grads = ab.Gaussians.zeros_like(r["theta"])
    ab.abcd_backward(ctx, r["theta"], r["cam"], None, r["proj"], r["tiles"], r["F"], r["B"],
                     r["fbd"], None, r["out"], r["state"], torch.from_numpy(gt).cuda(), 0.2, loss,
                     None, grads)
    ctx.sync()
    R = oracle.render(case.sp, case.off, case.ids, W, H, F=case.F64(), B=case.B64())
    L, dL = oracle.loss(R["out"][..., :3], gt.astype(np.float64), 0.2)
    g2 = oracle.backward(case.sp, case.off, case.ids, W, H, dL, F=case.F64(), B=case.B64())
    ref = oracle.project_backward(case.g, case.cam, g2)
    return loss.item(), L, grads, ref, R, gt, r


def test_train_step_matches_separate_calls(ctx, tiny):
    """abcd_train_step (the six entry points of a step in one call) gives the same loss and,
    up to the order of the backward's atomic sums, the same parameters and Adam moments as
    calling project, bin_sort, render, backward and Adam one by one."""
    case = Case(tiny, 1, fb=True)
    H, W = case.cam.height, case.cam.width
    cam = ab.camera(case.cam)
    gt = torch.from_numpy(sg.random_image(H, W, 3, seed=77)).cuda()
    F = torch.from_numpy(case.F).cuda()
    B = torch.from_numpy(case.B).cuda()
    lr = [1e-3, 5e-3, 1e-3, 0.025, 2.5e-3, 1.25e-4]
    res = []
    for fused in (False, True):
        theta = ab.Gaussians.from_numpy(case.g)
        grads, m, v = (ab.Gaussians.zeros_like(theta) for _ in range(3))
        proj = ab.Projected.alloc(theta.n)
        tiles = ab.Tiles.alloc(1_000_000, W, H)
        out = torch.empty(H, W, 4, device="cuda")
        st = ab.FwdState.alloc(W, H)
        loss = torch.zeros(2, device="cuda")
        step = ab.TrainStep(ctx, theta, grads, m, v, proj, tiles, out, st, lr)
        for k in range(2):
            if fused:
                step(cam, F, B, gt, loss[k:k + 1], k + 1)
            else:
                ab.abcd_project(ctx, theta, cam, None, proj)
                ab.abcd_bin_sort(ctx, proj, theta.n, cam, tiles)
                ab.abcd_render_composite_fwd(ctx, cam, None, proj, tiles, F, B, ab.ABCD_F16, None,
                                             out, st)
                ab.abcd_backward(ctx, theta, cam, None, proj, tiles, F, B, ab.ABCD_F16, None, out,
                                 st, gt, 0.2, loss[k:k + 1], None, grads)
                ab.abcd_adam_active(ctx, theta, grads, m, v, lr, 0.9, 0.999, 1e-15, k + 1)
        ctx.sync()
        res.append((loss.cpu(), [t.cpu() for t in theta.tensors() + m.tensors() + v.tensors()]))
    assert torch.equal(res[0][0][:1], res[1][0][:1])            # first loss: same inputs
    assert torch.allclose(res[0][0], res[1][0], rtol=1e-5, atol=0)
    for a_, b_ in zip(res[0][1], res[1][1]):
        assert torch.allclose(a_, b_, rtol=1e-4, atol=1e-7)


@pytest.mark.parametrize("seed,cam_idx", [(1001, 0), (1005, 1)])
def test_full_step_matches_oracle(ctx, seed, cam_idx):
    """project -> bin/sort -> render + composite -> L1 + 0.2 D-SSIM -> backward, element-wise.
    The seeded configurations have no decision within fp32 reach of its threshold (asserted),
    so every parameter gradient is compared strictly."""
    scene = sg.tiny_scene(seed=seed, per_cell=300, res=64, n_cams=4)
    case = Case(scene, cam_idx, fb=True)
    lg, L, grads, ref, R, _, _ = _full_step(ctx, scene, case)
    assert int((R["n_ev"] > 0).sum()) == 0 and not case.opt and not case.amb_r.any()
    assert abs(lg - L) <= 1e-5 * L
    for name, t in zip(("means", "log_scales", "quats", "opacity_logits", "sh"), grads.tensors()):
        # spec tolerance (1e-3 relative or 1e-5 absolute), with the absolute floor taken
        # as 1e-5 of the group's largest gradient when that is smaller
        atol = min(1e-5, 1e-5 * float(np.abs(ref[name]).max()))
        par.assert_grad_close(t.cpu().numpy(), ref[name], rtol=1e-3, atol=atol, what=name)


def test_full_step_tiny_scene(ctx, tiny):
    """The 2x2x2 x 2,000 workload at 128x128: loss to 1e-5; every gradient group to 1e-3 in
    relative L2 norm; and element-wise at the benchmark spec's tolerance with the loss gradient zeroed,
    on both sides, within 10 pixels (the reach of the SSIM windows' coupling) of every pixel
    holding a decision within fp32 rounding of its threshold, so that no such pixel feeds
    either gradient."""
    from scipy import ndimage
    case = Case(tiny, 1, fb=True)
    lg, L, grads, ref, R, gt, r = _full_step(ctx, tiny, case)
    assert abs(lg - L) <= 1e-5 * L
    for name, t in zip(GROUPS, grads.tensors()):
        got = t.cpu().numpy().astype(np.float64)
        rel = np.linalg.norm(got - ref[name]) / max(np.linalg.norm(ref[name]), 1e-30)
        assert rel < 1e-3, (name, rel)
    W, H = case.cam.width, case.cam.height
    bad = (R["n_ev"] > 0) | par.opt_pixel_mask(case.P, case.opt, case.cam)
    keep = ~ndimage.binary_dilation(bad, structure=np.ones((21, 21), bool))
    print(f"tiny-scene step: {bad.sum()} pixels with an ambiguous decision, {keep.mean():.0%} kept")
    assert keep.mean() > 0.3
    _, dL = oracle.loss(R["out"][..., :3], gt.astype(np.float64), 0.2)
    g2 = oracle.backward(case.sp, case.off, case.ids, W, H, dL * keep[..., None], F=case.F64(),
                         B=case.B64())
    refm = oracle.project_backward(case.g, case.cam, g2)
    loss = torch.zeros(1, device="cuda")
    dl = torch.empty(H, W, 3, device="cuda")
    ab.abcd_loss(ctx, r["out"], torch.from_numpy(gt).cuda(), W, H, 0.2, loss, dl)
    dl *= torch.from_numpy(keep.astype(np.float32)).cuda()[..., None]
    grad2d = torch.empty(r["theta"].n, 9, device="cuda")
    ab.abcd_render_backward(ctx, r["cam"], None, r["proj"], r["tiles"], r["F"], r["B"], r["fbd"],
                            None, r["state"], dl, r["theta"].n, grad2d)
    gm = ab.Gaussians.zeros_like(r["theta"])
    ab.abcd_project_backward(ctx, r["theta"], r["cam"], None, grad2d, gm)
    ctx.sync()
    for name, t in zip(GROUPS, gm.tensors()):
        atol = min(1e-5, 1e-5 * float(np.abs(refm[name]).max()))
        par.assert_grad_close(t.cpu().numpy(), refm[name], rtol=1e-3, atol=atol,
                              what=f"{name} (kept pixels)")


def test_capacity_overflow_reported(ctx, tiny):
    case = Case(tiny, 0, fb=False)
    cam = ab.camera(case.cam)
    theta = ab.Gaussians.from_numpy(case.g)
    proj = ab.Projected.alloc(theta.n)
    ab.abcd_project(ctx, theta, cam, None, proj)
    tiles = ab.Tiles.alloc(100, case.cam.width, case.cam.height)
    ab.abcd_bin_sort(ctx, proj, theta.n, cam, tiles)
    with pytest.raises(ab.AbcdError) as ei:
        ctx.sync()
    assert ei.value.status == ab.ABCD_ERR_CAPACITY
    assert abs(int(tiles.count.item()) - len(case.ids)) <= sum(len(v) for v in case.opt_list.values())
    assert int(tiles.ranges.abs().sum().item()) == 0
    ctx.clear_status()
    ctx.sync()


def test_bin_sort_wait_timeout_reported(ctx):
    """The radix sort's look-back waits are bounded: with tile 0 of the depth sort's first pass
    withheld (a test hook: it publishes nothing) and a short wait limit, the tiles behind it give
    up, abcd_sync reports ABCD_ERR_TIMEOUT and the call returns; once the status is cleared the
    same context sorts correctly again.  A render queued behind the timed-out sort reads every
    list as empty (the lists may hold stale ids): its image is the empty one."""
    s = sg.grid_scene((1, 1, 1), 5.0, 6000, 0, seed=97)
    s.cameras = sg.ring_cameras(1, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 96, 64, seed=97)
    g = s.gaussians
    assert g.n > 2 * 2048             # the depth sort's passes span three look-back tiles
    cam = ab.camera(s.cameras[0])
    theta = ab.Gaussians.from_numpy(g)
    proj = ab.Projected.alloc(theta.n)
    ab.abcd_project(ctx, theta, cam, None, proj)
    tiles = ab.Tiles.alloc(1 << 20, s.cameras[0].width, s.cameras[0].height)
    ab.abcd_bin_sort(ctx, proj, theta.n, cam, tiles)
    ctx.sync()
    K = int(tiles.count.item())
    ref_ids = tiles.ids[:K].clone()
    ref_rng = tiles.ranges.clone()
    L = ab.lib()
    assert L.abcd_set_wait_limit(ctx.h, 256) == ab.ABCD_OK
    assert L.abcd_test_withhold_lookback(ctx.h, 0) == ab.ABCD_OK
    ab.abcd_bin_sort(ctx, proj, theta.n, cam, tiles)
    H, W = s.cameras[0].height, s.cameras[0].width
    out = torch.full((H, W, 4), 7.0, device="cuda")
    ab.abcd_render_composite_fwd(ctx, cam, None, proj, tiles, None, None, ab.ABCD_F16, None, out,
                                 None)
    with pytest.raises(ab.AbcdError) as ei:
        ctx.sync()
    assert ei.value.status == ab.ABCD_ERR_TIMEOUT
    assert torch.count_nonzero(out).item() == 0
    ctx.clear_status()
    assert L.abcd_set_wait_limit(ctx.h, 1 << 20) == ab.ABCD_OK
    ab.abcd_bin_sort(ctx, proj, theta.n, cam, tiles)
    ctx.sync()
    assert int(tiles.count.item()) == K
    assert torch.equal(tiles.ids[:K], ref_ids) and torch.equal(tiles.ranges, ref_rng)


def test_invalid_arguments_rejected(ctx):
    cam = ab.abcd_camera()
    cam.width = 0
    theta = ab.Gaussians(*(torch.zeros(1, k, device="cuda") for k in (3, 3, 4, 1, 3)), 0)
    theta.opacity_logits = torch.zeros(1, device="cuda")
    with pytest.raises(ab.AbcdError) as ei:
        ab.abcd_project(ctx, theta, cam, None, ab.Projected.alloc(1))
    assert ei.value.status == ab.ABCD_ERR_INVALID_ARG
