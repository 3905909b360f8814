"""CPU oracle for the ABCD active-block step -- TEST INFRASTRUCTURE ONLY.

Plain fp64 C++ (``abcd_oracle.cpp``) behind ctypes, with numpy-friendly wrappers.  It is
what the CUDA path is checked against; it shares no code with it.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may import it.

Parity unpinned: none of the functions here (each is pinned by tests/test_oracle_pins.py).
Only reported, not pinned: the difference between the partition-layered render and a single
global depth sort of every Gaussian.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liborc.so")
_SRC = os.path.join(_HERE, "abcd_oracle.cpp")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (C++17, -O2, no FP contraction, OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH) or
             os.path.getmtime(_LIB_PATH) < max(os.path.getmtime(_SRC),
                                               os.path.getmtime(os.path.join(_HERE, "abcd_oracle.h"))))
    if force or stale:
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        cmd = ["g++", "-std=c++17", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-fopenmp",
               "-fno-fast-math", "-o", tmp, _SRC]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class Camera(C.Structure):
    _fields_ = [("R", C.c_double * 9), ("t", C.c_double * 3), ("fx", C.c_double),
                ("fy", C.c_double), ("cx", C.c_double), ("cy", C.c_double),
                ("width", C.c_int), ("height", C.c_int)]


class Opts(C.Structure):
    _fields_ = [("near_z", C.c_double), ("dilation", C.c_double), ("guard", C.c_double),
                ("alpha_max", C.c_double), ("alpha_min", C.c_double), ("t_min", C.c_double),
                ("tile", C.c_int)]


class Gaussians(C.Structure):
    _fields_ = [("means", C.c_void_p), ("log_scales", C.c_void_p), ("quats", C.c_void_p),
                ("opacity_logits", C.c_void_p), ("sh", C.c_void_p), ("n", C.c_int),
                ("sh_degree", C.c_int)]


class Projected(C.Structure):
    _fields_ = [(k, C.c_void_p) for k in ("visible", "depth", "depth_key", "uv", "conic",
                                          "opacity", "rgb", "rgb_raw", "eig", "radius_exact",
                                          "radius", "rect", "view_tan")]


class Splats(C.Structure):
    _fields_ = [("n", C.c_int), ("uv", C.c_void_p), ("conic", C.c_void_p),
                ("opacity", C.c_void_p), ("rgb", C.c_void_p)]


class Margins(C.Structure):
    _fields_ = [("m_uv", C.c_void_p), ("m_conic", C.c_void_p), ("k_arith", C.c_double),
                ("eps_alpha", C.c_double), ("eps_step", C.c_double)]


EV_SKIP, EV_TERM, EV_CLAMP = 1, 2, 3


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = C.CDLL(build())
            _lib.orc_tile_lists.restype = C.c_longlong
            _lib.orc_box_min_sigma.restype = C.c_double
            _lib.orc_box_min_sigma.argtypes = [C.c_void_p, C.c_double, C.c_double, C.c_double,
                                               C.c_double]
            _lib.orc_sh_basis.restype = C.c_double
            _lib.orc_sh_basis.argtypes = [C.c_int, C.c_int, C.c_double, C.c_double, C.c_double]
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _f64(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def default_opts(**over) -> Opts:
    o = Opts()
    lib().orc_default_opts(C.byref(o))
    for k, v in over.items():
        setattr(o, k, v)
    return o


def camera(cam) -> Camera:
    """Convert a scenegen.Camera (float32 values) to the oracle's fp64 camera, exactly."""
    c = Camera()
    c.R[:] = [float(x) for x in np.asarray(cam.R, dtype=np.float64).reshape(-1)]
    c.t[:] = [float(x) for x in np.asarray(cam.t, dtype=np.float64).reshape(-1)]
    c.fx, c.fy, c.cx, c.cy = float(cam.fx), float(cam.fy), float(cam.cx), float(cam.cy)
    c.width, c.height = int(cam.width), int(cam.height)
    return c


class _GaussKeep:
    """Holds fp64 copies of the parameters alive while the C struct points at them."""

    def __init__(self, g):
        self.means = _f64(g.means)
        self.log_scales = _f64(g.log_scales)
        self.quats = _f64(g.quats)
        self.logits = _f64(g.opacity_logits)
        self.sh = _f64(g.sh)
        self.n = int(self.means.shape[0])
        self.deg = int(g.sh_degree)
        self.s = Gaussians(_p(self.means), _p(self.log_scales), _p(self.quats),
                           _p(self.logits), _p(self.sh), self.n, self.deg)


def project(g, cam, opts=None) -> dict:
    """Per-Gaussian projection (dict of numpy arrays, fp64 unless integer)."""
    opts = opts or default_opts()
    k = _GaussKeep(g)
    n = k.n
    out = dict(visible=np.zeros(n, np.int32), depth=np.zeros(n), depth_key=np.zeros(n, np.uint32),
               uv=np.zeros((n, 2)), conic=np.zeros((n, 3)), opacity=np.zeros(n),
               rgb=np.zeros((n, 3)), rgb_raw=np.zeros((n, 3)), eig=np.zeros((n, 2)),
               radius_exact=np.zeros(n), radius=np.zeros(n, np.int32),
               rect=np.zeros((n, 4), np.int32), view_tan=np.zeros((n, 2)))
    P = Projected(*[_p(out[f]) for f, _ in Projected._fields_])
    rc = lib().orc_project(C.byref(k.s), C.byref(camera(cam)), C.byref(opts), C.byref(P))
    assert rc == 0
    return out


def project_backward(g, cam, grad2d, opts=None) -> dict:
    opts = opts or default_opts()
    k = _GaussKeep(g)
    n, D = k.n, (k.deg + 1) ** 2
    g2 = _f64(grad2d).reshape(n, 9)
    out = dict(means=np.zeros((n, 3)), log_scales=np.zeros((n, 3)), quats=np.zeros((n, 4)),
               opacity_logits=np.zeros(n), sh=np.zeros((n, D, 3)))
    rc = lib().orc_project_backward(C.byref(k.s), C.byref(camera(cam)), C.byref(opts), _p(g2),
                                    _p(out["means"]), _p(out["log_scales"]), _p(out["quats"]),
                                    _p(out["opacity_logits"]), _p(out["sh"]))
    assert rc == 0
    return out


def tiles_xy(width, height, tile=16):
    return (width + tile - 1) // tile, (height + tile - 1) // tile


# The renderer's listing reading (R1b): a tile is listed when the least sigma over its pixel
# centres, in log2 units, is at most (thr (1 + LIST_REL) + LIST_ABS) (1 + LIST_REL), thr =
# log2(opacity / alpha_min): the exact rule widened by a margin that keeps every tile the exact
# rule keeps whatever the fp32 rounding of the extent computation.
LIST_REL = 1e-3
LIST_ABS = 0.01


def tile_lists(proj, width, height, tile=16, rule="listing", alpha_min=1.0 / 255.0):
    """Returns (offsets[n_tiles + 1] int64, ids[K] int32).  rule="listing" (the renderer's
    listing rule, R1b) keeps a tile of the 3-sigma square where the least sigma over its pixel
    centres is within the margin above ln(o / alpha_min); rule="alpha" keeps exactly the tiles
    on which the Gaussian can reach alpha_min; rule="square" keeps the whole square (3DGS)."""
    assert rule in ("listing", "alpha", "square"), rule
    tx, ty = tiles_xy(width, height, tile)
    vis = np.ascontiguousarray(proj["visible"], dtype=np.int32)
    rect = np.ascontiguousarray(proj["rect"], dtype=np.int32)
    key = np.ascontiguousarray(proj["depth_key"], dtype=np.uint32)
    n = vis.shape[0]
    cap = int(np.sum(vis * np.maximum(rect[:, 2] - rect[:, 0], 0) *
                     np.maximum(rect[:, 3] - rect[:, 1], 0)))
    offsets = np.zeros(tx * ty + 1, np.int64)
    ids = np.zeros(max(cap, 1), np.int32)
    sp = SplatSet.from_proj(proj) if rule != "square" else None
    rel, ab_ = (LIST_REL, LIST_ABS) if rule == "listing" else (0.0, 0.0)
    K = lib().orc_tile_lists(n, _p(vis), _p(rect), _p(key), tx, ty, _p(offsets), _p(ids),
                             C.c_longlong(cap), C.byref(sp.s) if sp is not None else None,
                             C.c_double(alpha_min), int(tile), C.c_double(rel), C.c_double(ab_))
    assert 0 <= K <= cap, (K, cap)
    return offsets, ids[:K]


def box_min_sigma(conic, X0, X1, Y0, Y1):
    q = _f64(conic)
    return lib().orc_box_min_sigma(_p(q), float(X0), float(X1), float(Y0), float(Y1))


class SplatSet:
    """Screen-space splats (+ optional event margins) kept alive for the C calls."""

    def __init__(self, uv, conic, opacity, rgb, m_uv=None, m_conic=None, k_arith=0.0,
                 eps_alpha=0.0, eps_step=0.0):
        self.uv, self.conic, self.opacity, self.rgb = _f64(uv), _f64(conic), _f64(opacity), _f64(rgb)
        self.s = Splats(int(self.uv.shape[0]), _p(self.uv), _p(self.conic), _p(self.opacity),
                        _p(self.rgb))
        self.mg = None
        if m_uv is not None:
            self.m_uv, self.m_conic = _f64(m_uv), _f64(m_conic)
            self.mg = Margins(_p(self.m_uv), _p(self.m_conic), float(k_arith), float(eps_alpha),
                              float(eps_step))

    @classmethod
    def from_proj(cls, proj, **kw):
        return cls(proj["uv"], proj["conic"], proj["opacity"], proj["rgb"], **kw)


def _img(a, H, W, ch=4):
    return None if a is None else _f64(a).reshape(H, W, ch)


def render(splats: SplatSet, offsets, ids, width, height, F=None, B=None, bg=None, opts=None,
           max_ev=4):
    """Whole image. Returns dict(out[H,W,4], A[H,W,4], T_final[H,W], n_used[H,W], ev, n_ev)."""
    opts = opts or default_opts()
    H, W = height, width
    offsets = np.ascontiguousarray(offsets, dtype=np.int64)
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    F, B = _img(F, H, W), _img(B, H, W)
    bgv = None if bg is None else _f64(bg)
    out = np.zeros((H, W, 4)); A = np.zeros((H, W, 4)); Tf = np.zeros((H, W))
    nu = np.zeros((H, W), np.int32)
    ev = np.zeros((H, W, max_ev, 2), np.int32); nev = np.zeros((H, W), np.int32)
    rc = lib().orc_render_image(C.byref(splats.s), _p(offsets), _p(ids), W, H, C.byref(opts),
                                _p(F), _p(B), _p(bgv),
                                C.byref(splats.mg) if splats.mg is not None else None,
                                _p(out), _p(A), _p(Tf), _p(nu), _p(ev), max_ev, _p(nev))
    assert rc == 0
    return dict(out=out, A=A, T_final=Tf, n_used=nu, ev=ev, n_ev=nev)


def render_pixel(splats: SplatSet, lst, px, py, F=None, B=None, bg=None, toggles=(), opts=None,
                 max_ev=8):
    opts = opts or default_opts()
    lst = np.ascontiguousarray(lst, dtype=np.int32)
    tg = np.ascontiguousarray(np.asarray(toggles, dtype=np.int32).reshape(-1, 2))
    out4, A4 = np.zeros(4), np.zeros(4)
    Tf, nu, nev = C.c_double(), C.c_int(), C.c_int()
    ev = np.zeros((max_ev, 2), np.int32)
    Fp = None if F is None else _f64(F)
    Bp = None if B is None else _f64(B)
    bgv = None if bg is None else _f64(bg)
    lib().orc_render_pixel(C.byref(splats.s), _p(lst), int(lst.shape[0]), int(px), int(py),
                           C.byref(opts), _p(Fp), _p(Bp), _p(bgv), _p(tg), int(tg.shape[0]),
                           C.byref(splats.mg) if splats.mg is not None else None,
                           _p(out4), _p(A4), C.byref(Tf), C.byref(nu), _p(ev), max_ev,
                           C.byref(nev))
    return dict(out=out4, A=A4, T_final=Tf.value, n_used=nu.value,
                events=[tuple(e) for e in ev[:min(nev.value, max_ev)]], n_ev=nev.value)


def backward_pixel(splats: SplatSet, lst, px, py, G, F=None, B=None, bg=None, toggles=(),
                   opts=None, grad2d=None):
    opts = opts or default_opts()
    lst = np.ascontiguousarray(lst, dtype=np.int32)
    tg = np.ascontiguousarray(np.asarray(toggles, dtype=np.int32).reshape(-1, 2))
    if grad2d is None:
        grad2d = np.zeros((splats.s.n, 9))
    Fp = None if F is None else _f64(F)
    Bp = None if B is None else _f64(B)
    bgv = None if bg is None else _f64(bg)
    Gv = _f64(G)
    lib().orc_backward_pixel(C.byref(splats.s), _p(lst), int(lst.shape[0]), int(px), int(py),
                             C.byref(opts), _p(Fp), _p(Bp), _p(bgv), _p(tg), int(tg.shape[0]),
                             _p(Gv), _p(grad2d))
    return grad2d


def backward(splats: SplatSet, offsets, ids, width, height, G, F=None, B=None, bg=None,
             opts=None):
    """grad2d[n, 9] = dL/d(u, v, a, b, c, opacity, r, g, b) given G = dL/d(final rgb)."""
    opts = opts or default_opts()
    H, W = height, width
    offsets = np.ascontiguousarray(offsets, dtype=np.int64)
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    F, B = _img(F, H, W), _img(B, H, W)
    bgv = None if bg is None else _f64(bg)
    Gv = _img(G, H, W, 3)
    grad2d = np.zeros((splats.s.n, 9))
    rc = lib().orc_backward_image(C.byref(splats.s), _p(offsets), _p(ids), W, H, C.byref(opts),
                                  _p(F), _p(B), _p(bgv), _p(Gv), _p(grad2d))
    assert rc == 0
    return grad2d


def backward_pixels(splats: SplatSet, offsets, ids, width, height, G, pixels, F=None, B=None,
                    bg=None, opts=None):
    """backward() over the listed pixels only (linear indices): equal to it when G vanishes
    at every other pixel (each pixel's terms carry a factor of G)."""
    opts = opts or default_opts()
    H, W = height, width
    offsets = np.ascontiguousarray(offsets, dtype=np.int64)
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    F, B = _img(F, H, W), _img(B, H, W)
    bgv = None if bg is None else _f64(bg)
    Gv = _img(G, H, W, 3)
    pix = np.ascontiguousarray(np.sort(np.asarray(pixels, dtype=np.int64)), dtype=np.int32)
    grad2d = np.zeros((splats.s.n, 9))
    rc = lib().orc_backward_pixels(C.byref(splats.s), _p(offsets), _p(ids), W, H, C.byref(opts),
                                   _p(F), _p(B), _p(bgv), _p(Gv), _p(pix), int(pix.shape[0]),
                                   _p(grad2d))
    assert rc == 0
    return grad2d


def composite_layers(layers, order):
    """Left fold of 'over' over layers[order[k]]; layers [L, H, W, 4] -> [H, W, 4]."""
    layers = _f64(layers)
    L, H, W, _ = layers.shape
    order = np.ascontiguousarray(order, dtype=np.int32)
    out = np.zeros((H, W, 4))
    lib().orc_composite_layers(H * W, _p(layers), _p(order), int(order.shape[0]), _p(out))
    return out


def layer_visibility(layers, order):
    """(visible[L], coverage[L]) of layers [L, H, W, 4] taken in `order` (front to back)."""
    layers = _f64(layers)
    L, H, W, _ = layers.shape
    order = np.ascontiguousarray(order, dtype=np.int32)
    vis, cov = np.zeros(L), np.zeros(L)
    rc = lib().orc_layer_visibility(H * W, L, _p(layers), _p(order), int(order.shape[0]),
                                    _p(vis), _p(cov))
    assert rc == 0, "repeated or out-of-range layer index"
    return vis, cov


def loss(x, y, lam, with_grad=True):
    x, y = _f64(x), _f64(y)
    H, W, _ = x.shape
    val = C.c_double()
    grad = np.zeros_like(x) if with_grad else None
    lib().orc_loss(W, H, _p(x), _p(y), C.c_double(lam), C.byref(val), _p(grad))
    return val.value, grad


def ssim_map(x, y):
    x, y = _f64(x), _f64(y)
    H, W, _ = x.shape
    m = np.zeros_like(x)
    lib().orc_ssim_map(W, H, _p(x), _p(y), _p(m))
    return m


def adam(theta, grad, m, v, lr, beta1, beta2, eps, step):
    """In place on fp64 arrays."""
    for a in (theta, m, v):
        assert a.dtype == np.float64 and a.flags.c_contiguous
    g = _f64(grad)
    lib().orc_adam(C.c_longlong(theta.size), _p(theta), _p(g), _p(m), _p(v), C.c_double(lr),
                   C.c_double(beta1), C.c_double(beta2), C.c_double(eps), int(step))


def assign_cells(means, origin, side, dims):
    means = _f64(means)
    n = means.shape[0]
    cell = np.zeros(n, np.int32)
    o = _f64(origin)
    d = np.ascontiguousarray(dims, dtype=np.int32)
    lib().orc_assign_cells(n, _p(means), _p(o), C.c_double(side), _p(d), _p(cell))
    return cell


def partition_split(dims, origin, side, campos, active):
    d = np.ascontiguousarray(dims, dtype=np.int32)
    n = int(np.prod(d))
    front, back = np.zeros(n, np.int32), np.zeros(n, np.int32)
    nf, nb = C.c_int(), C.c_int()
    rc = lib().orc_partition_split(_p(d), _p(_f64(origin)), C.c_double(side), _p(_f64(campos)),
                                   int(active), _p(front), C.byref(nf), _p(back), C.byref(nb))
    assert rc == 0
    return front[:nf.value].copy(), back[:nb.value].copy()


def block_bounds(g) -> np.ndarray:
    """Box (lowest x, y, z, highest x, y, z) of the Gaussians' 3-sigma ellipsoids."""
    k = _GaussKeep(g)
    box = np.zeros(6)
    assert lib().orc_block_bounds(C.byref(k.s), _p(box)) == 0
    return box


def pair_visible(cam, box, opts=None) -> bool:
    opts = opts or default_opts()
    b = _f64(box)
    v = C.c_int()
    assert lib().orc_pair_visible(C.byref(camera(cam)), C.byref(opts), _p(b), C.byref(v)) == 0
    return bool(v.value)


def sh_basis(l, m, x, y, z):
    return lib().orc_sh_basis(l, m, x, y, z)


def cpu_threads() -> int:
    """Threads the oracle's OpenMP loops use (OMP_NUM_THREADS, else the affinity set)."""
    env = os.environ.get("OMP_NUM_THREADS")
    if env:
        try:
            return max(1, int(env.split(",")[0]))
        except ValueError:
            pass
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1
