"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test pins one part of the oracle to something other than itself: a closed form of the
EWA splat for one Gaussian, scipy's spherical harmonics, brute-force tile scans, central
finite differences in fp64, torch's Adam, the associativity of 'over' (Section 2), and a
ray-sampled depth order of grid cells.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2608_27735_gb300 import scenegen as sg


def make_gaussians(means, log_scales, quats, logits, sh, deg):
    return sg.Gaussians(np.asarray(means, np.float32).reshape(-1, 3),
                        np.asarray(log_scales, np.float32).reshape(-1, 3),
                        np.asarray(quats, np.float32).reshape(-1, 4),
                        np.asarray(logits, np.float32).reshape(-1),
                        np.asarray(sh, np.float32).reshape(len(np.asarray(logits).reshape(-1)),
                                                           (deg + 1) ** 2, 3), deg)


def identity_camera(W, H, f):
    return sg.Camera(R=np.eye(3, dtype=np.float32), t=np.zeros(3, np.float32), fx=f, fy=f,
                     cx=W / 2.0, cy=H / 2.0, width=W, height=H)


def render_scene(g, cam, opts=None, F=None, B=None, bg=None):
    P = oracle.project(g, cam, opts)
    off, ids = oracle.tile_lists(P, cam.width, cam.height)
    return P, off, ids, oracle.render(oracle.SplatSet.from_proj(P), off, ids, cam.width,
                                      cam.height, F=F, B=B, bg=bg, opts=opts)


# ----------------------------------------------------------------------------------------
# Single-Gaussian closed form (3DGS EWA splat, camera = identity)

@pytest.mark.parametrize("x0,y0,z0,s,sh0,logit", [
    (0.0, 0.0, 4.0, 0.05, 0.3, 0.4),
    (0.3, -0.2, 5.0, 0.08, -0.5, 1.2),
    (2.8, 0.3, 4.0, 0.5, 0.2, 0.1),      # off-screen mean: x/z beyond 1.3 tan(fov/2)
])
def test_single_gaussian_closed_form(x0, y0, z0, s, sh0, logit):
    W = H = 64
    f = 70.0
    g = make_gaussians([x0, y0, z0], [math.log(s)] * 3, [1, 0, 0, 0], [logit],
                       [sh0, sh0 * 0.5, -sh0], 0)
    cam = identity_camera(W, H, f)
    P, off, ids, R = render_scene(g, cam)
    x0, y0, z0 = (float(np.float32(v)) for v in (x0, y0, z0))
    s2 = float(np.exp(np.float64(np.float32(math.log(s))))) ** 2
    # Sigma' = s^2 J J^T + 0.3 I with J = [[f/z, 0, -f x'/z^2], [0, f/z, -f y'/z^2]], where
    # x' = z * clamp(x/z, +-1.3 tan(fov_x/2)) (3DGS frustum guard), likewise y'
    lim = 1.3 * (W / 2.0) / f
    xg, yg = z0 * np.clip(x0 / z0, -lim, lim), z0 * np.clip(y0 / z0, -lim, lim)
    J = np.array([[f / z0, 0, -f * xg / z0 ** 2], [0, f / z0, -f * yg / z0 ** 2]])
    S2 = s2 * J @ J.T + 0.3 * np.eye(2)
    Q = np.linalg.inv(S2)
    u, v = f * x0 / z0 + W / 2.0, f * y0 / z0 + H / 2.0
    o = 1.0 / (1.0 + math.exp(-float(np.float32(logit))))
    c0 = 1.0 / (2.0 * math.sqrt(math.pi))      # Y_00
    col = np.maximum(0.0, c0 * np.array([sh0, sh0 * 0.5, -sh0], np.float32).astype(np.float64) + 0.5)
    lam = np.linalg.eigvalsh(S2)
    mid, disc = lam.mean(), ((lam[1] - lam[0]) / 2) ** 2
    r = math.ceil(3 * math.sqrt(mid + math.sqrt(max(0.1, disc))))
    assert P["radius"][0] == r
    np.testing.assert_allclose(P["uv"][0], [u, v], rtol=0, atol=1e-12)
    np.testing.assert_allclose(P["conic"][0], [Q[0, 0], Q[0, 1], Q[1, 1]], rtol=1e-12)
    ys, xs = np.mgrid[0:H, 0:W]
    d = np.stack([xs + 0.5 - u, ys + 0.5 - v], -1)
    sig = 0.5 * np.einsum("...i,ij,...j->...", d, Q, d)
    alpha = np.minimum(0.99, o * np.exp(-sig))
    in_rect = ((xs // 16 >= max(0, math.floor((u - r) / 16))) & (xs // 16 <= math.floor((u + r) / 16)) &
               (ys // 16 >= max(0, math.floor((v - r) / 16))) & (ys // 16 <= math.floor((v + r) / 16)))
    alpha = np.where((alpha >= 1 / 255) & in_rect, alpha, 0.0)
    np.testing.assert_allclose(R["out"][..., 3], alpha, atol=1e-12)
    np.testing.assert_allclose(R["out"][..., :3], alpha[..., None] * col, atol=1e-12)
    np.testing.assert_allclose(R["T_final"], 1 - alpha, atol=1e-12)


def test_rotation_of_scale_axes():
    """A 90 degree turn about z swaps the x and y scales of the world covariance."""
    W = H = 64
    f = 60.0
    a = math.sqrt(0.5)
    base = dict(means=[0.1, 0.05, 4.0], logits=[0.0], sh=[0.2, 0.1, 0.0], deg=0)
    g1 = make_gaussians(base["means"], [math.log(0.2), math.log(0.05), math.log(0.1)],
                        [a, 0, 0, a], base["logits"], base["sh"], 0)
    g2 = make_gaussians(base["means"], [math.log(0.05), math.log(0.2), math.log(0.1)],
                        [1, 0, 0, 0], base["logits"], base["sh"], 0)
    cam = identity_camera(W, H, f)
    P1, P2 = oracle.project(g1, cam), oracle.project(g2, cam)
    np.testing.assert_allclose(P1["conic"], P2["conic"], rtol=1e-6)
    # unnormalised quaternion gives the same result
    g3 = make_gaussians(base["means"], [math.log(0.2), math.log(0.05), math.log(0.1)],
                        [3 * a, 0, 0, 3 * a], base["logits"], base["sh"], 0)
    np.testing.assert_allclose(oracle.project(g3, cam)["conic"], P1["conic"], rtol=1e-12)


def test_rigid_motion_invariance_deg0():
    """Moving camera and scene by the same rigid motion leaves the image unchanged."""
    s = sg.tiny_scene(per_cell=40, res=48, n_cams=1)
    g, cam = s.gaussians, s.cameras[0]
    _, _, _, R0 = render_scene(g, cam)
    rng = np.random.default_rng(3)
    q = rng.normal(size=4); q /= np.linalg.norm(q)
    w, x, y, z = q
    Rm = np.array([[1 - 2 * (y * y + z * z), 2 * (x * y - w * z), 2 * (x * z + w * y)],
                   [2 * (x * y + w * z), 1 - 2 * (x * x + z * z), 2 * (y * z - w * x)],
                   [2 * (x * z - w * y), 2 * (y * z + w * x), 1 - 2 * (x * x + y * y)]])
    tr = rng.normal(size=3)
    g2 = g.subset(slice(None))
    g2.means = (g.means.astype(np.float64) @ Rm.T + tr)
    qq = g.quats.astype(np.float64)
    # quaternion product q * q_i rotates each Gaussian's frame by Rm
    w2 = w * qq[:, 0] - x * qq[:, 1] - y * qq[:, 2] - z * qq[:, 3]
    x2 = w * qq[:, 1] + x * qq[:, 0] + y * qq[:, 3] - z * qq[:, 2]
    y2 = w * qq[:, 2] - x * qq[:, 3] + y * qq[:, 0] + z * qq[:, 1]
    z2 = w * qq[:, 3] + x * qq[:, 2] - y * qq[:, 1] + z * qq[:, 0]
    g2.quats = np.stack([w2, x2, y2, z2], -1)
    cam2 = sg.Camera(R=cam.R.astype(np.float64) @ Rm.T, t=cam.t.astype(np.float64) - cam.R.astype(np.float64) @ Rm.T @ tr,
                     fx=cam.fx, fy=cam.fy, cx=cam.cx, cy=cam.cy, width=cam.width, height=cam.height)

    class G64:   # keep fp64 values (the oracle reads fp64)
        pass
    g64 = G64()
    g64.means, g64.log_scales, g64.quats = g2.means, g.log_scales, g2.quats
    g64.opacity_logits, g64.sh, g64.sh_degree = g.opacity_logits, g.sh, 0
    P2 = oracle.project(g64, cam2)
    P1 = oracle.project(g, cam)
    np.testing.assert_array_equal(P1["visible"], P2["visible"])
    v = P1["visible"] == 1
    np.testing.assert_allclose(P2["uv"][v], P1["uv"][v], atol=1e-8)
    np.testing.assert_allclose(P2["conic"][v], P1["conic"][v], rtol=1e-7, atol=1e-10)
    np.testing.assert_allclose(P2["rgb"][v], P1["rgb"][v], atol=1e-12)


# ----------------------------------------------------------------------------------------
# Spherical harmonics

def test_sh_matches_scipy_and_known_constants():
    sp = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(0)
    dirs = rng.normal(size=(20, 3))
    dirs /= np.linalg.norm(dirs, axis=1, keepdims=True)
    assert abs(oracle.sh_basis(0, 0, 0, 0, 1) - 0.28209479177387814) < 1e-15
    assert abs(oracle.sh_basis(1, -1, 0, 1, 0) + 0.4886025119029199) < 1e-14
    for x, y, z in dirs:
        theta, phi = math.acos(z), math.atan2(y, x)
        for l in range(4):
            for m in range(-l, l + 1):
                Yc = sp.sph_harm_y(l, abs(m), theta, phi)     # includes Condon-Shortley phase
                ref = Yc.real if m == 0 else math.sqrt(2) * (Yc.real if m > 0 else Yc.imag)
                assert abs(oracle.sh_basis(l, m, x, y, z) - ref) < 1e-12, (l, m)


def test_sh_orthonormal_by_quadrature():
    # Gauss-Legendre in cos(theta) x uniform in phi: exact for polynomials of degree <= 6
    xs, ws = np.polynomial.legendre.leggauss(12)
    phis = 2 * np.pi * (np.arange(24) + 0.5) / 24
    idx = [(l, m) for l in range(4) for m in range(-l, l + 1)]
    G = np.zeros((16, 16))
    for z, wz in zip(xs, ws):
        st = math.sqrt(1 - z * z)
        for ph in phis:
            d = (st * math.cos(ph), st * math.sin(ph), z)
            Y = np.array([oracle.sh_basis(l, m, *d) for l, m in idx])
            G += wz * (2 * np.pi / 24) * np.outer(Y, Y)
    np.testing.assert_allclose(G, np.eye(16), atol=1e-12)


# ----------------------------------------------------------------------------------------
# Binning / sort

def test_tile_lists_brute_force():
    s = sg.tiny_scene(per_cell=60, res=80, n_cams=1)
    cam = s.cameras[0]
    P = oracle.project(s.gaussians, cam)
    off, ids = oracle.tile_lists(P, cam.width, cam.height, rule="square")
    tx, ty = oracle.tiles_xy(cam.width, cam.height)
    n = s.gaussians.n
    assert P["visible"].sum() > 0
    for t in range(tx * ty):
        bx, by = t % tx, t // tx
        members = []
        for i in range(n):
            if P["depth"][i] <= 0.2:
                continue
            u, v = P["uv"][i]
            r = P["radius"][i]
            # the square [u-r, u+r] x [v-r, v+r] meets the tile box [16 bx, 16 bx + 16) x ...
            if u - r < 16 * bx + 16 and u + r >= 16 * bx and v - r < 16 * by + 16 and v + r >= 16 * by:
                members.append(i)
        members.sort(key=lambda i: (int(P["depth_key"][i]), i))
        assert list(ids[off[t]:off[t + 1]]) == members, t
    # depth key is the fp32 depth, order-preserving as an unsigned integer
    vis = P["visible"] == 1
    z32 = P["depth_key"][vis].view(np.float32)
    assert np.all(np.abs(z32.astype(np.float64) - P["depth"][vis]) <= 4e-7 * P["depth"][vis])


@pytest.mark.parametrize("rule", ["alpha", "listing"])
def test_alpha_listing_rule_drops_only_skipped_entries(rule):
    """The alpha rule keeps a tile of the 3-sigma square only where the Gaussian can reach
    alpha_min, and the renderer's listing rule (R1b) only where it comes within the listing
    margin of that: every dropped entry is skipped by all 256 pixel centres of its tile, and the
    rendered image is bit-identical to the one over the full squares."""
    s = sg.tiny_scene(per_cell=300, res=96, n_cams=2)
    for cam in s.cameras:
        P = oracle.project(s.gaussians, cam)
        oq, iq = oracle.tile_lists(P, cam.width, cam.height, rule="square")
        oa, ia = oracle.tile_lists(P, cam.width, cam.height, rule=rule)
        tx, ty = oracle.tiles_xy(cam.width, cam.height)
        assert len(ia) < len(iq)
        ys, xs = np.mgrid[0:16, 0:16] + 0.5
        for t in range(tx * ty):
            full = list(iq[oq[t]:oq[t + 1]])
            kept = list(ia[oa[t]:oa[t + 1]])
            assert [g for g in full if g in set(kept)] == kept, t
            for g in set(full) - set(kept):
                u, v = P["uv"][g]
                a, b, c = P["conic"][g]
                dx, dy = xs + 16 * (t % tx) - u, ys + 16 * (t // tx) - v
                sig = 0.5 * (a * dx * dx + c * dy * dy) + b * dx * dy
                assert np.all(P["opacity"][g] * np.exp(-sig) < 1 / 255), (t, g)
        sp = oracle.SplatSet.from_proj(P)
        Rq = oracle.render(sp, oq, iq, cam.width, cam.height)
        Ra = oracle.render(sp, oa, ia, cam.width, cam.height)
        np.testing.assert_array_equal(Ra["out"], Rq["out"])
        np.testing.assert_array_equal(Ra["T_final"], Rq["T_final"])


def test_listing_margin_keeps_a_superset_of_the_alpha_rule():
    """The listing rule's lists hold the alpha rule's in the same order; an entry it adds has
    its least sigma over the tile's pixel centres above ln(o / alpha_min) (no pixel of the tile
    reaches alpha_min) and at most the margin's limit, and the margin adds few entries."""
    s = sg.tiny_scene(per_cell=600, res=128, n_cams=3)
    for cam in s.cameras:
        P = oracle.project(s.gaussians, cam)
        oa, ia = oracle.tile_lists(P, cam.width, cam.height, rule="alpha")
        ol, il = oracle.tile_lists(P, cam.width, cam.height, rule="listing")
        tx, ty = oracle.tiles_xy(cam.width, cam.height)
        extra = 0
        for t in range(tx * ty):
            kept = list(ia[oa[t]:oa[t + 1]])
            listed = list(il[ol[t]:ol[t + 1]])
            assert [g for g in listed if g in set(kept)] == kept, t
            x, y = t % tx, t // tx
            for g in set(listed) - set(kept):
                extra += 1
                u, v = P["uv"][g]
                m = oracle.box_min_sigma(P["conic"][g], 16 * x + 0.5 - u, 16 * x + 15.5 - u,
                                         16 * y + 0.5 - v, 16 * y + 15.5 - v)
                thr = math.log(P["opacity"][g] * 255.0)
                lim = (thr / math.log(2) * (1 + oracle.LIST_REL) + oracle.LIST_ABS) * \
                    (1 + oracle.LIST_REL) * math.log(2)
                assert thr < m <= lim, (t, g, m, thr, lim)
        assert len(il) == len(ia) + extra
        assert extra <= 0.02 * len(ia), (extra, len(ia))


def test_box_min_sigma_against_dense_sampling():
    rng = np.random.default_rng(21)
    for _ in range(300):
        L = rng.normal(size=(2, 2))
        S = L @ L.T + 0.3 * np.eye(2)
        Q = np.linalg.inv(S) * rng.uniform(0.01, 3.0)
        conic = [Q[0, 0], Q[0, 1], Q[1, 1]]
        X0, Y0 = rng.uniform(-30, 30, 2)
        X1, Y1 = X0 + rng.uniform(0, 15), Y0 + rng.uniform(0, 15)
        m = oracle.box_min_sigma(conic, X0, X1, Y0, Y1)
        gx, gy = np.meshgrid(np.linspace(X0, X1, 401), np.linspace(Y0, Y1, 401))
        sig = 0.5 * (Q[0, 0] * gx * gx + Q[1, 1] * gy * gy) + Q[0, 1] * gx * gy
        dense = sig.min()
        h = max(X1 - X0, Y1 - Y0) / 400
        grad = np.abs(Q).sum() * (max(abs(X0), abs(X1)) + max(abs(Y0), abs(Y1)))
        assert m <= dense + 1e-12
        assert dense - m <= grad * h + 1e-12
    assert oracle.box_min_sigma([1.0, 0.2, 2.0], -1, 1, -3, 2) == 0.0


def test_tile_lists_capacity_report():
    s = sg.tiny_scene(per_cell=10, res=48, n_cams=1)
    P = oracle.project(s.gaussians, s.cameras[0])
    off, ids = oracle.tile_lists(P, 48, 48, rule="square")
    import ctypes as C
    K = len(ids)
    o2 = np.zeros_like(off)
    i2 = np.zeros(max(K, 1), np.int32)
    r = oracle.lib().orc_tile_lists(P["visible"].shape[0], oracle._p(P["visible"]),
                                    oracle._p(P["rect"]), oracle._p(P["depth_key"]), 3, 3,
                                    oracle._p(o2), oracle._p(i2), C.c_longlong(K - 1), None,
                                    C.c_double(1 / 255), 16)
    assert r == -K - 1


# ----------------------------------------------------------------------------------------
# Render invariants and the compositing identity (Section 2)

def test_render_invariants_tiny_scene():
    s = sg.tiny_scene()
    cam = s.cameras[0]
    _, _, _, R = render_scene(s.gaussians, cam)
    out, A, Tf = R["out"], R["A"], R["T_final"]
    assert np.all((Tf >= 1e-4) & (Tf <= 1.0))
    np.testing.assert_allclose(A[..., 3], 1 - Tf, atol=1e-15)
    assert np.all((out[..., 3] >= 0) & (out[..., 3] <= 1))
    assert np.all(A[..., :3] <= (1 - Tf)[..., None] + 1e-12)   # colours lie in [0, 1]
    assert np.all(A[..., :3] >= 0)
    assert (R["n_used"] > 0).mean() > 0.3


def test_backward_over_a_pixel_list_equals_the_full_backward():
    """The restricted backward (the sampled full-size tests use it) is the full one when the
    upstream gradient vanishes off the list: every term of a pixel carries a factor of G."""
    s = sg.tiny_scene()
    cam = s.cameras[2]
    g = s.gaussians.subset(slice(0, 3000))
    P = oracle.project(g, cam)
    off, ids = oracle.tile_lists(P, cam.width, cam.height)
    sp = oracle.SplatSet.from_proj(P)
    rng = np.random.default_rng(12)
    pix = rng.choice(cam.width * cam.height, 900, replace=False)
    G = np.zeros((cam.height, cam.width, 3))
    G.reshape(-1, 3)[pix] = rng.normal(size=(900, 3))
    F = sg.premultiplied_layers(2, cam.height, cam.width, seed=4).astype(np.float64)
    full = oracle.backward(sp, off, ids, cam.width, cam.height, G, F=F[0], B=F[1])
    part = oracle.backward_pixels(sp, off, ids, cam.width, cam.height, G, pix, F=F[0], B=F[1])
    assert np.abs(full).max() > 0
    np.testing.assert_array_equal(part, full)


def _layer_lists(P, cells, part_order, tx, ty):
    """Per-tile lists of the explicit render of the given partitions, layered in order."""
    per = []
    for p in part_order:
        Pp = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in P.items()}
        Pp["visible"] = np.where(cells == p, P["visible"], 0).astype(np.int32)
        per.append(oracle.tile_lists(Pp, tx * 16, ty * 16))
    off = np.zeros(tx * ty + 1, np.int64)
    ids = []
    for t in range(tx * ty):
        for o_, i_ in per:
            ids.extend(i_[o_[t]:o_[t + 1]])
        off[t + 1] = len(ids)
    return off, np.asarray(ids, np.int32)


@pytest.mark.parametrize("t_min", [0.0, 1e-4])
def test_composited_equals_explicit_render(t_min):
    """Rendering every partition explicitly (partition-layered) equals F over A over B."""
    s = sg.tiny_scene(res=64, per_cell=500)
    g = s.gaussians
    cells = oracle.assign_cells(g.means, s.grid.origin, s.grid.side, s.grid.dims)
    opts = oracle.default_opts(t_min=t_min)
    for ci, cam in enumerate(s.cameras[:2]):
        for active in (0, 5):
            front, back = oracle.partition_split(s.grid.dims, s.grid.origin, s.grid.side,
                                                 cam.position, active)
            P = oracle.project(g, cam, opts)
            tx, ty = oracle.tiles_xy(64, 64)
            sp = oracle.SplatSet.from_proj(P)
            layers = {}
            for p in list(front) + list(back) + [active]:
                o_, i_ = _layer_lists(P, cells, [p], tx, ty)
                layers[p] = oracle.render(sp, o_, i_, 64, 64, opts=opts)["out"]
            stack = np.stack([layers[p] for p in range(8)])
            F = oracle.composite_layers(stack, front)
            B = oracle.composite_layers(stack, back)
            o_a, i_a = _layer_lists(P, cells, [active], tx, ty)
            comp = oracle.render(sp, o_a, i_a, 64, 64, F=F, B=B, opts=opts)["out"]
            o_all, i_all = _layer_lists(P, cells, list(front) + [active] + list(back), tx, ty)
            explicit = oracle.render(sp, o_all, i_all, 64, 64, opts=opts)["out"]
            err = np.abs(comp - explicit).max()
            if t_min == 0.0:
                assert err < 1e-12, (ci, active, err)
            else:   # early termination differs per layer: bounded by t_min / (1 - alpha_max)
                assert err <= 1e-4 / (1 - 0.99) + 1e-12, (ci, active, err)
            # split invariance: any split point gives the same composite of all layers
            full = oracle.composite_layers(stack, list(front) + [active] + list(back))
            Fs = oracle.composite_layers(stack, front)
            mid = oracle.composite_layers(stack, [active] + list(back))
            assert np.abs(Fs + (1 - Fs[..., 3:]) * mid - full).max() < 1e-13


def test_over_constant_layers_golden():
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "over_constant_layers.txt")
    layers, expect = [], None
    for line in open(path):
        if line.startswith("layer"):
            layers.append([float(v) for v in line.split()[1:]])
        elif line.startswith("expect"):
            expect = [float(v) for v in line.split()[1:]]
    st = np.array(layers)[:, None, None, :]
    out = oracle.composite_layers(st, [0, 1, 2])
    np.testing.assert_array_equal(out[0, 0], expect)


def _premultiplied_layers(rng, L, H, W, clear=0.3):
    """Random premultiplied RGBA layers (colour <= alpha), each with a share of clear pixels."""
    a = rng.uniform(0, 1, (L, H, W, 1)) * (rng.uniform(0, 1, (L, H, W, 1)) > clear)
    return np.concatenate([a * rng.uniform(0, 1, (L, H, W, 3)), a], -1)


def test_visibility_constant_layers_closed_form():
    """Constant alphas 0.5, 0.25, 0.8 taken in the order 2, 0, 1: each layer's visible share is
    its alpha times the transmittance of the layers before it, worked by hand."""
    alphas = [0.5, 0.25, 0.8]
    st = np.stack([np.full((3, 5, 4), a) for a in alphas])
    vis, cov = oracle.layer_visibility(st, [2, 0, 1])
    np.testing.assert_allclose(cov, alphas, rtol=0, atol=1e-15)
    np.testing.assert_allclose(vis, [0.5 * 0.2, 0.25 * 0.2 * 0.5, 0.8], rtol=0, atol=1e-15)
    # a layer left out of the order has neither; an opaque layer hides everything behind it
    vis, cov = oracle.layer_visibility(st, [1])
    np.testing.assert_allclose(vis, [0, 0.25, 0], atol=1e-15)
    np.testing.assert_allclose(cov, [0, 0.25, 0], atol=1e-15)
    opaque = np.concatenate([st, np.ones((1, 3, 5, 4))])
    vis, cov = oracle.layer_visibility(opaque, [3, 0, 1, 2])
    np.testing.assert_allclose(vis, [0, 0, 0, 1], atol=1e-15)
    np.testing.assert_allclose(cov, alphas + [1.0], atol=1e-15)


def test_visibility_telescopes_to_the_composite_alpha():
    """1 - prod(1 - a_k) = sum_k a_k prod_{i<k} (1 - a_i): the visible shares of all layers add
    up to the mean alpha of their composite (checked against composite_layers)."""
    rng = np.random.default_rng(11)
    st = _premultiplied_layers(rng, 7, 9, 13)
    for order in ([0, 1, 2, 3, 4, 5, 6], [6, 2, 4, 0, 5, 1, 3], [3, 1, 5]):
        vis, cov = oracle.layer_visibility(st, order)
        comp = oracle.composite_layers(st, order)
        assert abs(vis.sum() - comp[..., 3].mean()) < 1e-13, order
        np.testing.assert_allclose(cov[order], st[order][..., 3].mean(axis=(1, 2)), atol=1e-15)
        assert np.all(vis <= cov + 1e-15)


def test_culling_error_bound():
    """Leaving a set D of layers out of the composite changes every channel of every pixel by
    at most sum_{j in D} a_j T_j when colours are premultiplied and at most alpha: the mean
    error of the culled composite is at most the sum of the dropped layers' visible shares."""
    rng = np.random.default_rng(12)
    st = _premultiplied_layers(rng, 6, 11, 10)
    order = [4, 0, 5, 2, 1, 3]
    vis, _ = oracle.layer_visibility(st, order)
    full = oracle.composite_layers(st, order)
    for drop in ({0}, {4}, {3}, {0, 2}, {4, 5, 1}, set(order)):
        kept = [j for j in order if j not in drop]
        culled = oracle.composite_layers(st, kept) if kept else np.zeros_like(full)
        err = np.abs(full - culled).mean(axis=(0, 1))
        bound = sum(vis[j] for j in drop)
        assert np.all(err <= bound + 1e-13), (drop, err, bound)
        if drop == set(order):          # nothing kept: the alpha error is the bound exactly
            assert abs(err[3] - bound) < 1e-13


def test_bg_and_fb_in_closed_form():
    """Empty active block: out = F over B (+ (1 - out.a) bg)."""
    rng = np.random.default_rng(1)
    H = W = 16
    Fa = rng.uniform(0, 1, (H, W, 1)); F = np.concatenate([Fa * rng.uniform(0, 1, (H, W, 3)), Fa], -1)
    Ba = rng.uniform(0, 1, (H, W, 1)); B = np.concatenate([Ba * rng.uniform(0, 1, (H, W, 3)), Ba], -1)
    bg = np.array([0.2, 0.3, 0.4])
    sp = oracle.SplatSet(np.zeros((1, 2)), np.zeros((1, 3)), np.zeros(1), np.zeros((1, 3)))
    R = oracle.render(sp, np.zeros(2, np.int64), np.zeros(0, np.int32), W, H, F=F, B=B, bg=bg)
    a = F[..., 3:] + (1 - F[..., 3:]) * B[..., 3:]
    rgb = F[..., :3] + (1 - F[..., 3:]) * B[..., :3] + (1 - a) * bg
    np.testing.assert_allclose(R["out"][..., :3], rgb, atol=1e-15)
    np.testing.assert_allclose(R["out"][..., 3:], a, atol=1e-15)


# ----------------------------------------------------------------------------------------
# Finite differences (fp64) of the whole chain: params -> projection -> blend -> composite

def _fd_setup(seed, deg=3, n=6, W=32, H=16):
    rng = np.random.default_rng(seed)
    means = np.c_[rng.uniform(-0.4, 0.4, n), rng.uniform(-0.2, 0.2, n), rng.uniform(3.0, 4.0, n)]
    means[0] = [2.3, 0.0, 3.0]          # off-screen mean: exercises the guard clamp in J
    ls = np.log(rng.uniform(0.15, 0.35, (n, 3)))
    ls[0] = np.log([0.9, 0.9, 0.9])
    q = rng.normal(size=(n, 4))
    logits = rng.uniform(-1.5, 1.0, n)
    D = (deg + 1) ** 2
    sh = rng.normal(0, 0.1, (n, D, 3))
    sh[:, 0, :] = rng.uniform(0.5, 1.5, (n, 3))     # keep colours away from the clamp at 0
    g = sg.Gaussians(means, ls, q, logits, sh, deg)   # fp64 arrays: the oracle reads fp64
    cam = identity_camera(W, H, 30.0)
    Fa = rng.uniform(0.1, 0.6, (H, W, 1)); F = np.concatenate([Fa * rng.uniform(0, 1, (H, W, 3)), Fa], -1)
    Ba = rng.uniform(0.2, 0.9, (H, W, 1)); B = np.concatenate([Ba * rng.uniform(0, 1, (H, W, 3)), Ba], -1)
    G = rng.normal(size=(H, W, 3))
    bg = np.array([0.3, 0.1, 0.7])
    return g, cam, F, B, G, bg


def _objective(g, cam, F, B, G, bg, opts):
    P = oracle.project(g, cam, opts)
    assert np.all(P["rect"][P["visible"] == 1] == [0, 0, 2, 1]), "rect must cover both tiles"
    off, ids = oracle.tile_lists(P, cam.width, cam.height)
    R = oracle.render(oracle.SplatSet.from_proj(P), off, ids, cam.width, cam.height,
                      F=F, B=B, bg=bg, opts=opts)
    return float(np.sum(G * R["out"][..., :3])), P, off, ids


def test_gradient_matches_finite_differences():
    g, cam, F, B, G, bg = _fd_setup(5)
    # smooth regime: no alpha skip, no early stop (their branches have zero derivative)
    opts = oracle.default_opts(alpha_min=0.0, t_min=0.0)
    f0, P, off, ids = _objective(g, cam, F, B, G, bg, opts)
    assert abs(P["view_tan"][0, 0]) > 1.3 * (cam.width / 2 / cam.fx)   # guard active
    assert np.all(P["rgb_raw"] > 0.05)
    g2d = oracle.backward(oracle.SplatSet.from_proj(P), off, ids, cam.width, cam.height, G,
                          F=F, B=B, bg=bg, opts=opts)
    grads = oracle.project_backward(g, cam, g2d, opts)
    worst = 0.0
    for name in ("means", "log_scales", "quats", "opacity_logits", "sh"):
        arr = getattr(g, name)
        flat = arr.reshape(-1)
        ana = grads[name].reshape(-1)
        for k in range(flat.size):
            h = 1e-6 * max(1.0, abs(flat[k]))
            old = flat[k]
            flat[k] = old + h; fp = _objective(g, cam, F, B, G, bg, opts)[0]
            flat[k] = old - h; fm = _objective(g, cam, F, B, G, bg, opts)[0]
            flat[k] = old
            fd = (fp - fm) / (2 * h)
            err = abs(fd - ana[k]) / max(1e-3, abs(fd), abs(ana[k]))
            worst = max(worst, err)
            assert err < 1e-5, (name, k, fd, ana[k])
    assert worst < 1e-5


def test_gradient_alpha_clamp_is_flat():
    """An opacity driven past the 0.99 clamp has zero opacity gradient at its centre pixel."""
    g, cam, F, B, G, bg = _fd_setup(6, deg=0, n=1)
    g.means[0] = [0.0, 0.0, 3.0]
    g.log_scales[0] = np.log([1.0, 1.0, 1.0])
    g.opacity_logits[0] = 8.0
    opts = oracle.default_opts(alpha_min=0.0, t_min=0.0)
    f0, P, off, ids = _objective(g, cam, F, B, G, bg, opts)
    sp = oracle.SplatSet.from_proj(P)
    u, v = P["uv"][0]
    px, py = int(u), int(v)
    g2 = oracle.backward_pixel(sp, ids[off[0]:off[1]] if px < 16 else ids[off[1]:off[2]], px, py,
                               G[py, px], F=F[py, px], B=B[py, px], bg=bg, opts=opts)
    assert g2[0, 5] == 0.0 and g2[0, 0] == 0.0
    assert g2[0, 6] != 0.0


# ----------------------------------------------------------------------------------------
# Loss

def test_ssim_identity_and_scipy_window():
    ndi = pytest.importorskip("scipy.ndimage")
    rng = np.random.default_rng(2)
    x = rng.uniform(0, 1, (20, 27, 3))
    y = np.clip(x + rng.normal(0, 0.1, x.shape), 0, 1)
    assert abs(oracle.loss(x, x, 1.0, with_grad=False)[0]) < 1e-14
    np.testing.assert_allclose(oracle.ssim_map(x, x), 1.0, atol=1e-14)
    # SSIM map via scipy's 2-D correlation with the outer-product window, zero padding
    g1 = np.exp(-((np.arange(11) - 5.0) ** 2) / (2 * 1.5 ** 2)); g1 /= g1.sum()
    w = np.outer(g1, g1)
    ref = np.zeros_like(x)
    for c in range(3):
        f = lambda a: ndi.correlate(a, w, mode="constant", cval=0.0)
        mx, my = f(x[..., c]), f(y[..., c])
        vx, vy = f(x[..., c] ** 2) - mx ** 2, f(y[..., c] ** 2) - my ** 2
        cxy = f(x[..., c] * y[..., c]) - mx * my
        ref[..., c] = ((2 * mx * my + 1e-4) * (2 * cxy + 9e-4)) / ((mx ** 2 + my ** 2 + 1e-4) * (vx + vy + 9e-4))
    np.testing.assert_allclose(oracle.ssim_map(x, y), ref, atol=1e-13)
    L, _ = oracle.loss(x, y, 0.2, with_grad=False)
    np.testing.assert_allclose(L, 0.8 * np.abs(x - y).mean() + 0.2 * (1 - ref.mean()), rtol=1e-13)


def test_loss_gradient_finite_differences():
    rng = np.random.default_rng(4)
    x = rng.uniform(0, 1, (9, 13, 3))
    y = rng.uniform(0, 1, (9, 13, 3))
    _, gr = oracle.loss(x, y, 0.2)
    for k in rng.choice(x.size, 60, replace=False):
        xp = x.copy().reshape(-1); xm = x.copy().reshape(-1)
        xp[k] += 1e-6; xm[k] -= 1e-6
        fd = (oracle.loss(xp.reshape(x.shape), y, 0.2, False)[0] -
              oracle.loss(xm.reshape(x.shape), y, 0.2, False)[0]) / 2e-6
        assert abs(fd - gr.reshape(-1)[k]) <= 1e-7 * max(1.0, abs(fd)) + 1e-9


# ----------------------------------------------------------------------------------------
# Adam

def test_adam_first_step_closed_form_and_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(7)
    th = rng.normal(size=50); g1 = rng.normal(size=50); g2 = rng.normal(size=50)
    m = np.zeros(50); v = np.zeros(50); t = th.copy()
    oracle.adam(t, g1, m, v, 0.01, 0.9, 0.999, 1e-15, 1)
    np.testing.assert_allclose(t, th - 0.01 * g1 / (np.abs(g1) + 1e-15), rtol=0, atol=1e-15)
    oracle.adam(t, g2, m, v, 0.01, 0.9, 0.999, 1e-15, 2)
    p = torch.nn.Parameter(torch.tensor(th, dtype=torch.float64))
    opt = torch.optim.Adam([p], lr=0.01, betas=(0.9, 0.999), eps=1e-15)
    for gg in (g1, g2):
        p.grad = torch.tensor(gg, dtype=torch.float64)
        opt.step()
    np.testing.assert_allclose(t, p.detach().numpy(), rtol=0, atol=1e-14)


# ----------------------------------------------------------------------------------------
# Partitions: assignment by mean and per-camera depth order (Section 2, Section 4)

def test_assign_cells_by_mean():
    s = sg.tiny_scene(per_cell=50)
    cells = oracle.assign_cells(s.gaussians.means, s.grid.origin, s.grid.side, s.grid.dims)
    np.testing.assert_array_equal(cells, s.block_of)


def test_partition_split_ties_go_back_golden():
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "partition_split_ties.txt")
    for line in open(path):
        if not line.strip() or line.startswith("#"):
            continue
        f = line.split("|")
        dims = [int(v) for v in f[0].split()]
        campos = [float(v) for v in f[1].split()]
        active = int(f[2])
        front = [int(v) for v in f[3].split()]
        back = [int(v) for v in f[4].split()]
        fr, bk = oracle.partition_split(dims, np.zeros(3), 1.0, campos, active)
        assert list(fr) == front and list(bk) == back, line


def test_partition_order_consistent_with_rays():
    rng = np.random.default_rng(11)
    dims, side = (3, 3, 2), 5.0
    origin = -0.5 * side * np.array(dims, dtype=np.float64)
    lo, hi = origin, origin + side * np.array(dims)
    for trial in range(6):
        campos = rng.uniform(lo - 8, hi + 8)
        if trial == 0:
            campos = origin + side * np.array([1.5, 1.5, 0.5])   # inside cell (1, 1, 0)
        active = int(rng.integers(0, 18)) if trial else 4
        front, back = oracle.partition_split(dims, origin, side, campos, active)
        if trial == 0:
            assert len(front) == 0
        assert sorted(list(front) + list(back) + [active]) == list(range(18))
        fset = set(int(f) for f in front)
        for _ in range(1500):
            d = rng.normal(size=3); d /= np.linalg.norm(d)
            ts = np.linspace(0, 60, 3000)
            pts = campos + ts[:, None] * d
            idx = np.floor((pts - origin) / side).astype(int)
            ok = np.all((idx >= 0) & (idx < np.array(dims)), axis=1)
            seq = [int(i + dims[0] * (j + dims[1] * k)) for (i, j, k) in idx[ok]]
            if active not in seq:
                continue
            first_a = seq.index(active)
            for c in set(seq):
                if c == active:
                    continue
                if seq.index(c) < first_a:
                    assert c in fset, (campos, active, c)
                else:
                    assert c not in fset, (campos, active, c)


def test_blend_harness_form_equals_the_definition():
    """The oracle's test-harness form of the blend (event reporting under an uncertainty model,
    decisions inverted on request) gives, with no decision inverted, exactly the plain
    definition's image."""
    from tests import _parity as par
    s = sg.tiny_scene(per_cell=300, res=64, n_cams=2)
    for cam in s.cameras:
        P = oracle.project(s.gaussians, cam)
        off, ids = oracle.tile_lists(P, cam.width, cam.height)
        plain = oracle.render(oracle.SplatSet.from_proj(P), off, ids, cam.width, cam.height)
        probe = oracle.render(par.splats_with_margins(s.gaussians, cam, P), off, ids, cam.width,
                              cam.height)
        np.testing.assert_array_equal(plain["out"], probe["out"])
        np.testing.assert_array_equal(plain["T_final"], probe["T_final"])
        np.testing.assert_array_equal(plain["n_used"], probe["n_used"])


def _rot(q):
    w, x, y, z = np.asarray(q, np.float64) / np.linalg.norm(q)
    return np.array([[1 - 2 * (y * y + z * z), 2 * (x * y - w * z), 2 * (x * z + w * y)],
                     [2 * (x * y + w * z), 1 - 2 * (x * x + z * z), 2 * (y * z - w * x)],
                     [2 * (x * z - w * y), 2 * (y * z + w * x), 1 - 2 * (x * x + y * y)]])


def test_block_bounds_hold_every_3sigma_ellipsoid():
    """Points on every Gaussian's 3-sigma ellipsoid (mu + 3 R S u for unit u) lie in the box,
    and each face of the box is touched (up to the sampling) by one of them."""
    s = sg.grid_scene((1, 1, 1), 5.0, 40, 0, seed=61)
    g = s.gaussians
    box = oracle.block_bounds(g)
    rng = np.random.default_rng(3)
    u = rng.normal(size=(4000, 3))
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    pts = []
    for i in range(g.n):
        M = _rot(g.quats[i]) @ np.diag(np.exp(g.log_scales[i].astype(np.float64)))
        pts.append(g.means[i].astype(np.float64) + 3.0 * u @ M.T)
    pts = np.concatenate(pts)
    assert np.all(pts >= box[:3] - 1e-12) and np.all(pts <= box[3:] + 1e-12)
    span = box[3:] - box[:3]
    assert np.all(pts.min(0) - box[:3] <= 2e-2 * span) and np.all(box[3:] - pts.max(0) <= 2e-2 * span)


def test_pair_visibility_never_culls_a_seen_box():
    """Dense samples of random boxes: a box with a sample point inside the view frustum is
    always visible; a box reported not visible has every sample outside; closed-form cases."""
    cam = sg.look_at(np.array([0.0, -10.0, 0.0]), np.zeros(3), 160, 120)
    rng = np.random.default_rng(8)
    g = np.linspace(0.0, 1.0, 9)
    gx = 1.3 * 0.5 * cam.width / cam.fx
    gy = 1.3 * 0.5 * cam.height / cam.fy
    R, t = cam.R.astype(np.float64), cam.t.astype(np.float64)
    n_vis = n_cul = 0
    for _ in range(400):
        c = rng.uniform(-15, 15, 3)
        h = rng.uniform(0.2, 4.0, 3)
        box = np.concatenate([c - h, c + h])
        P = np.stack(np.meshgrid(g, g, g, indexing="ij"), -1).reshape(-1, 3)
        P = box[:3] + P * (box[3:] - box[:3])
        pc = P @ R.T + t
        inside = (pc[:, 2] >= 0.2) & (np.abs(pc[:, 0]) <= gx * pc[:, 2]) & \
            (np.abs(pc[:, 1]) <= gy * pc[:, 2])
        v = oracle.pair_visible(cam, box)
        if inside.any():
            assert v
        n_vis += v
        n_cul += not v
    assert n_vis > 50 and n_cul > 50
    pos = cam.position
    ahead = pos + 6.0 * (R.T @ np.array([0.0, 0.0, 1.0]))
    assert oracle.pair_visible(cam, np.concatenate([ahead - 0.1, ahead + 0.1]))
    behind = pos - 6.0 * (R.T @ np.array([0.0, 0.0, 1.0]))
    assert not oracle.pair_visible(cam, np.concatenate([behind - 0.1, behind + 0.1]))
    side = pos + 6.0 * (R.T @ np.array([0.0, 0.0, 1.0])) + 6.0 * gx * 1.5 * (R.T @ np.array([1.0, 0, 0]))
    assert not oracle.pair_visible(cam, np.concatenate([side - 0.1, side + 0.1]))
    assert not oracle.pair_visible(cam, np.array([1.0, 1.0, 1.0, 0.0, 0.0, 0.0]))   # empty


def test_culled_pairs_render_transparent():
    """Walk-through cameras inside a 4x4x2 grid: every camera-partition pair the rule culls
    lists no Gaussian on any tile in the oracle, so its layer is transparent (the reading loses
    nothing), and the rule culls a good share of the pairs."""
    s = sg.grid_scene((4, 4, 2), 5.0, 200, 0, seed=72)
    cams = sg.inside_cameras(s.grid, 8, 160, 107, seed=5)
    cells = oracle.assign_cells(s.gaussians.means, s.grid.origin, s.grid.side, s.grid.dims)
    culled = 0
    for cam in cams:
        for b in range(32):
            gb = s.gaussians.subset(np.nonzero(cells == b)[0])
            bx = oracle.block_bounds(gb)
            ijk = np.array([b % 4, (b // 4) % 4, b // 16], np.float64)
            lo = np.asarray(s.grid.origin) + s.grid.side * ijk
            box = np.concatenate([np.minimum(bx[:3], lo), np.maximum(bx[3:], lo + s.grid.side)])
            if oracle.pair_visible(cam, box):
                continue
            culled += 1
            P = oracle.project(gb, cam)
            off, ids = oracle.tile_lists(P, cam.width, cam.height)
            assert len(ids) == 0
    assert culled >= 0.3 * 32 * len(cams), culled
    print(f"culled pairs: {culled} of {32 * len(cams)}")
