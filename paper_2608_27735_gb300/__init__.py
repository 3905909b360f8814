"""GB300-native (sm_103a) ABCD active-block hot path.

The compute lives in ``libabcd.so`` (hand-written CUDA behind the C ABI declared in
``include/abcd.h``).  This module is the thin binding: ctypes structures mirroring the
header, functions with the same names (argument marshalling only), and small containers
that allocate the caller-owned device buffers with torch.  There is no CPU fallback: if the
library is missing or no GPU is present, every call raises.
"""
from __future__ import annotations

import ctypes as C
import os
import re
import threading
from dataclasses import dataclass

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libabcd.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "abcd.h")

ABCD_OK, ABCD_ERR_INVALID_ARG, ABCD_ERR_CUDA, ABCD_ERR_CAPACITY, ABCD_ERR_TIMEOUT, \
    ABCD_ERR_WORKSPACE = range(6)
ABCD_F16, ABCD_F32 = 0, 1
ABCD_MAX_CACHE_SLOTS = 4096
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "CUDA", 3: "CAPACITY", 4: "TIMEOUT", 5: "WORKSPACE"}
TILE = 16


class AbcdError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"abcd status {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


# ---------------------------------------------------------------------------------------
# ctypes mirrors of include/abcd.h

class abcd_camera(C.Structure):
    _fields_ = [("R", C.c_float * 9), ("t", C.c_float * 3), ("fx", C.c_float), ("fy", C.c_float),
                ("cx", C.c_float), ("cy", C.c_float), ("width", C.c_int), ("height", C.c_int)]


class abcd_render_opts(C.Structure):
    _fields_ = [(k, C.c_float) for k in ("near_z", "dilation", "guard", "alpha_max",
                                         "alpha_min", "t_min")]


class abcd_gaussians(C.Structure):
    _fields_ = [("means", C.c_void_p), ("log_scales", C.c_void_p), ("quats", C.c_void_p),
                ("opacity_logits", C.c_void_p), ("sh", C.c_void_p), ("n", C.c_int),
                ("sh_degree", C.c_int)]


class abcd_projected(C.Structure):
    _fields_ = [(k, C.c_void_p) for k in ("uv", "conic_opacity", "rgb", "depth", "radius",
                                          "tiles_touched")]


class abcd_tiles(C.Structure):
    _fields_ = [("ids", C.c_void_p), ("ranges", C.c_void_p), ("capacity", C.c_longlong),
                ("count", C.c_void_p)]


class abcd_fwd_state(C.Structure):
    _fields_ = [("A_T", C.c_void_p), ("n_last", C.c_void_p)]


class abcd_alu_peaks(C.Structure):
    _fields_ = [("sms", C.c_int), ("clock_mhz_nominal", C.c_double), ("ffma_tflops", C.c_double),
                ("ffma2_tflops", C.c_double), ("ex2_tops", C.c_double), ("ms_ffma", C.c_double),
                ("ms_ffma2", C.c_double), ("ms_ex2", C.c_double)]


_lock = threading.Lock()
_lib = None

_SIGS = {
    "abcd_create": [C.POINTER(C.c_void_p), C.c_int, C.c_void_p],
    "abcd_destroy": [C.c_void_p],
    "abcd_set_stream": [C.c_void_p, C.c_void_p],
    "abcd_workspace_size": [C.c_int, C.c_longlong, C.c_longlong, C.POINTER(C.c_size_t)],
    "abcd_set_workspace": [C.c_void_p, C.c_void_p, C.c_size_t, C.c_int, C.c_longlong, C.c_longlong],
    "abcd_sync": [C.c_void_p],
    "abcd_clear_status": [C.c_void_p],
    "abcd_project": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p],
    "abcd_bin_sort": [C.c_void_p, C.c_void_p, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p],
    "abcd_render_composite_fwd": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                  C.c_void_p, C.c_void_p, C.c_int, C.c_void_p, C.c_void_p,
                                  C.c_void_p, C.c_void_p],
    "abcd_loss": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_float, C.c_void_p,
                  C.c_void_p],
    "abcd_render_backward": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                             C.c_void_p, C.c_void_p, C.c_int, C.c_void_p, C.c_void_p,
                             C.c_void_p, C.c_int, C.c_void_p],
    "abcd_project_backward": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                              C.c_void_p],
    "abcd_backward": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                      C.c_void_p, C.c_void_p, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p,
                      C.c_void_p, C.c_float, C.c_void_p, C.c_void_p, C.c_void_p],
    "abcd_adam_active": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                         C.c_float, C.c_float, C.c_float, C.c_int],
    "abcd_composite_cache": [C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_void_p, C.c_int,
                             C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_int],
    "abcd_render_refresh_packed": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                   C.c_void_p, C.c_void_p, C.c_void_p],
    "abcd_composite_cache_packed": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_void_p,
                                    C.c_int, C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_int],
    "abcd_layer_visibility": [C.c_void_p, C.c_void_p, C.c_int, C.c_void_p, C.c_int, C.c_int,
                              C.c_int, C.c_void_p, C.c_void_p],
    "abcd_layer_visibility_packed": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_void_p,
                                     C.c_int, C.c_int, C.c_int, C.c_void_p, C.c_void_p],
    "abcd_train_step": [C.c_void_p] + [C.c_void_p] * 8 + [C.c_void_p, C.c_void_p, C.c_int,
                         C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_float, C.c_void_p,
                         C.c_void_p, C.c_float, C.c_float, C.c_float, C.c_int],
    "abcd_refresh_layer": [C.c_void_p] * 9,
    "abcd_cache_fetch": [C.c_void_p, C.c_int, C.c_void_p, C.c_void_p, C.c_size_t],
    "abcd_cache_wait": [C.c_void_p, C.c_int],
    "abcd_cache_release": [C.c_void_p, C.c_int],
    "abcd_cache_store": [C.c_void_p, C.c_int, C.c_void_p, C.c_void_p, C.c_size_t],
    "abcd_cache_sync": [C.c_void_p],
    "abcd_composite_fold_packed": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_int,
                                   C.c_void_p, C.c_void_p, C.c_void_p],
    "abcd_measure_alu_peaks": [C.c_int, C.c_void_p],
    "abcd_block_bounds": [C.c_void_p, C.c_void_p, C.c_void_p],
    "abcd_pair_visible": [C.c_void_p, C.c_void_p, C.c_void_p, C.POINTER(C.c_int)],
    "abcd_set_wait_limit": [C.c_void_p, C.c_uint],
    "abcd_test_withhold_lookback": [C.c_void_p, C.c_longlong],
    "abcd_assign_cells": [C.c_void_p, C.c_int, C.c_void_p, C.c_double, C.c_void_p, C.c_void_p],
    "abcd_partition_split": [C.c_void_p, C.c_void_p, C.c_double, C.c_void_p, C.c_int,
                             C.c_void_p, C.POINTER(C.c_int), C.c_void_p, C.POINTER(C.c_int)],
}


def build(force: bool = False) -> str:
    from . import _build
    return _build.build(force=force)


def lib():
    """The loaded libabcd.so.  Raises if it has not been built (no fallback)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"libabcd.so is not built ({LIB_PATH}); run "
                                   "paper_2608_27735_gb300.build() (nvcc, sm_103a)")
            L = C.CDLL(LIB_PATH)
            for name, args in _SIGS.items():
                f = getattr(L, name)
                f.argtypes = args
                f.restype = C.c_int
            L.abcd_last_error.argtypes = [C.c_void_p]
            L.abcd_last_error.restype = C.c_char_p
            L.abcd_launch_count.argtypes = [C.c_void_p]
            L.abcd_launch_count.restype = C.c_longlong
            _lib = L
    return _lib


def header_functions():
    """Names of the functions include/abcd.h declares."""
    txt = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:abcd_status|const char\*|long long)\s+(abcd_\w+)\s*\(",
                                 txt, flags=re.M)))


# ---------------------------------------------------------------------------------------
# device buffers (torch is the allocator; pointers only cross the ABI)

def _torch():
    import torch
    return torch


def _p(t):
    if t is None:
        return None
    assert t.is_cuda and t.is_contiguous(), "ABI arguments must be contiguous CUDA tensors"
    return C.c_void_p(t.data_ptr())


def _hp(t):
    assert (not t.is_cuda) and t.is_contiguous() and t.is_pinned(), \
        "host-tier buffers must be contiguous pinned host tensors"
    return C.c_void_p(t.data_ptr())


@dataclass
class Gaussians:
    """Active-block parameters (or gradients / Adam moments) as CUDA float32 tensors."""
    means: object
    log_scales: object
    quats: object
    opacity_logits: object
    sh: object
    sh_degree: int

    @property
    def n(self):
        return int(self.means.shape[0])

    def c(self):
        return abcd_gaussians(_p(self.means), _p(self.log_scales), _p(self.quats),
                              _p(self.opacity_logits), _p(self.sh), self.n, self.sh_degree)

    def tensors(self):
        return (self.means, self.log_scales, self.quats, self.opacity_logits, self.sh)

    @classmethod
    def from_numpy(cls, g, device="cuda"):
        torch = _torch()
        f = lambda a: torch.as_tensor(a, dtype=torch.float32).contiguous().to(device)
        return cls(f(g.means), f(g.log_scales), f(g.quats), f(g.opacity_logits), f(g.sh),
                   int(g.sh_degree))

    @classmethod
    def zeros_like(cls, o):
        torch = _torch()
        return cls(*(torch.zeros_like(t) for t in o.tensors()), o.sh_degree)


@dataclass
class Projected:
    uv: object
    conic_opacity: object
    rgb: object
    depth: object
    radius: object
    tiles_touched: object

    @classmethod
    def alloc(cls, n, device="cuda"):
        torch = _torch()
        f = lambda *s, dt=torch.float32: torch.empty(*s, dtype=dt, device=device)
        return cls(f(n, 2), f(n, 4), f(n, 3), f(n), f(n, dt=torch.int32), f(n, dt=torch.int32))

    def c(self):
        return abcd_projected(_p(self.uv), _p(self.conic_opacity), _p(self.rgb), _p(self.depth),
                              _p(self.radius), _p(self.tiles_touched))


@dataclass
class Tiles:
    ids: object
    ranges: object
    count: object
    capacity: int

    @classmethod
    def alloc(cls, capacity, width, height, device="cuda"):
        torch = _torch()
        nt = ((width + TILE - 1) // TILE) * ((height + TILE - 1) // TILE)
        return cls(torch.empty(max(1, capacity), dtype=torch.int32, device=device),
                   torch.zeros(nt, 2, dtype=torch.int32, device=device),
                   torch.zeros(1, dtype=torch.int64, device=device), int(capacity))

    def c(self):
        return abcd_tiles(_p(self.ids), _p(self.ranges), self.capacity, _p(self.count))


@dataclass
class FwdState:
    A_T: object
    n_last: object

    @classmethod
    def alloc(cls, width, height, device="cuda"):
        torch = _torch()
        return cls(torch.empty(height, width, 4, dtype=torch.float32, device=device),
                   torch.empty(height, width, dtype=torch.int32, device=device))

    def c(self):
        return abcd_fwd_state(_p(self.A_T), _p(self.n_last))


def camera(cam) -> abcd_camera:
    """abcd_camera from any object with R, t, fx, fy, cx, cy, width, height."""
    import numpy as np
    c = abcd_camera()
    c.R[:] = [float(v) for v in np.asarray(cam.R, dtype=np.float32).reshape(-1)]
    c.t[:] = [float(v) for v in np.asarray(cam.t, dtype=np.float32).reshape(-1)]
    c.fx, c.fy, c.cx, c.cy = float(cam.fx), float(cam.fy), float(cam.cx), float(cam.cy)
    c.width, c.height = int(cam.width), int(cam.height)
    return c


def render_opts(near_z=0.2, dilation=0.3, guard=1.3, alpha_max=0.99, alpha_min=1.0 / 255.0,
                t_min=1e-4) -> abcd_render_opts:
    return abcd_render_opts(near_z, dilation, guard, alpha_max, alpha_min, t_min)


class Context:
    """An abcd_ctx bound to a device and a CUDA stream, plus its caller-owned workspace."""

    def __init__(self, device=0, stream=None):
        torch = _torch()
        if not torch.cuda.is_available():
            raise RuntimeError("libabcd needs a CUDA device; there is no CPU fallback")
        self.device = device
        self.stream = stream if stream is not None else torch.cuda.current_stream(device)
        h = C.c_void_p()
        st = lib().abcd_create(C.byref(h), device, C.c_void_p(self.stream.cuda_stream))
        if st != ABCD_OK:
            raise AbcdError(st, "abcd_create failed")
        self.h = h
        self.workspace = None
        self.limits = (0, 0, 0)

    def __del__(self):
        try:
            if getattr(self, "h", None):
                lib().abcd_destroy(self.h)
                self.h = None
        except Exception:
            pass

    def check(self, st):
        if st != ABCD_OK:
            raise AbcdError(st, lib().abcd_last_error(self.h).decode(errors="replace"))

    def reserve(self, max_gaussians, max_pairs, max_pixels):
        """(Re)allocates the workspace if the limits grew."""
        torch = _torch()
        mg, mp, mx = (max(a, b) for a, b in zip((max_gaussians, max_pairs, max_pixels), self.limits))
        if self.workspace is not None and (mg, mp, mx) == self.limits:
            return
        nbytes = C.c_size_t()
        self.check(lib().abcd_workspace_size(mg, mp, mx, C.byref(nbytes)))
        ws = torch.empty(nbytes.value + 256, dtype=torch.uint8, device=self.device)
        off = (-ws.data_ptr()) % 256
        self.workspace = ws
        self.check(lib().abcd_set_workspace(self.h, C.c_void_p(ws.data_ptr() + off), nbytes.value,
                                            mg, mp, mx))
        self.limits = (mg, mp, mx)

    def sync(self):
        self.check(lib().abcd_sync(self.h))

    def clear_status(self):
        self.check(lib().abcd_clear_status(self.h))

    def launches(self):
        return int(lib().abcd_launch_count(self.h))


# ---------------------------------------------------------------------------------------
# the ABI, same names (each raises AbcdError on a non-OK status)

def _opt(o):
    return None if o is None else C.byref(o)


def abcd_project(ctx: Context, theta: Gaussians, cam: abcd_camera, opts, out: Projected):
    g = theta.c(); o = out.c()
    ctx.check(lib().abcd_project(ctx.h, C.byref(g), C.byref(cam), _opt(opts), C.byref(o)))


def abcd_bin_sort(ctx: Context, proj: Projected, n: int, cam: abcd_camera, out: Tiles,
                  opts=None):
    p = proj.c(); t = out.c()
    ctx.check(lib().abcd_bin_sort(ctx.h, C.byref(p), int(n), C.byref(cam), _opt(opts), C.byref(t)))


def _bg(bg):
    if bg is None:
        return None
    return (C.c_float * 3)(*[float(v) for v in bg])


def abcd_render_composite_fwd(ctx: Context, cam, opts, proj: Projected, tiles: Tiles, F=None,
                              B=None, fb_dtype=ABCD_F16, bg=None, out_rgba=None,
                              state: FwdState = None, refresh_f16=None):
    p = proj.c(); t = tiles.c()
    s = state.c() if state is not None else None
    ctx.check(lib().abcd_render_composite_fwd(
        ctx.h, C.byref(cam), _opt(opts), C.byref(p), C.byref(t), _p(F), _p(B), int(fb_dtype),
        _bg(bg), _p(out_rgba), C.byref(s) if s is not None else None, _p(refresh_f16)))


def abcd_loss(ctx: Context, out_rgba, gt_rgb, width, height, lambda_ssim, loss_out, dL_dout):
    ctx.check(lib().abcd_loss(ctx.h, _p(out_rgba), _p(gt_rgb), int(width), int(height),
                              float(lambda_ssim), _p(loss_out), _p(dL_dout)))


def abcd_render_backward(ctx: Context, cam, opts, proj: Projected, tiles: Tiles, F, B, fb_dtype,
                         bg, state: FwdState, dL_dout, n, grad2d):
    p = proj.c(); t = tiles.c(); s = state.c()
    ctx.check(lib().abcd_render_backward(ctx.h, C.byref(cam), _opt(opts), C.byref(p), C.byref(t),
                                         _p(F), _p(B), int(fb_dtype), _bg(bg), C.byref(s),
                                         _p(dL_dout), int(n), _p(grad2d)))


def abcd_project_backward(ctx: Context, theta: Gaussians, cam, opts, grad2d, grads: Gaussians):
    g = theta.c(); d = grads.c()
    ctx.check(lib().abcd_project_backward(ctx.h, C.byref(g), C.byref(cam), _opt(opts),
                                          _p(grad2d), C.byref(d)))


def abcd_backward(ctx: Context, theta: Gaussians, cam, opts, proj: Projected, tiles: Tiles, F, B,
                  fb_dtype, bg, out_rgba, state: FwdState, gt_rgb, lambda_ssim, loss_out,
                  dL_dout, grads: Gaussians):
    g = theta.c(); p = proj.c(); t = tiles.c(); s = state.c(); d = grads.c()
    ctx.check(lib().abcd_backward(ctx.h, C.byref(g), C.byref(cam), _opt(opts), C.byref(p),
                                  C.byref(t), _p(F), _p(B), int(fb_dtype), _bg(bg), _p(out_rgba),
                                  C.byref(s), _p(gt_rgb), float(lambda_ssim), _p(loss_out),
                                  _p(dL_dout), C.byref(d)))


def abcd_adam_active(ctx: Context, theta: Gaussians, grads: Gaussians, m: Gaussians, v: Gaussians,
                     lr, beta1, beta2, eps, step):
    a, g, mm, vv = theta.c(), grads.c(), m.c(), v.c()
    lrs = (C.c_float * 6)(*[float(x) for x in lr])
    ctx.check(lib().abcd_adam_active(ctx.h, C.byref(a), C.byref(g), C.byref(mm), C.byref(vv), lrs,
                                     float(beta1), float(beta2), float(eps), int(step)))


def abcd_composite_cache(ctx: Context, layers, order, split, width, height, F_out, B_out,
                         layer_dtype=ABCD_F16, out_dtype=ABCD_F16):
    """layers: list of CUDA tensors (or None at the active position); order: list of ints."""
    L = len(layers)
    arr = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in layers])
    ordr = (C.c_int * max(1, L))(*[int(k) for k in order])
    ctx.check(lib().abcd_composite_cache(ctx.h, arr, L, int(layer_dtype), ordr, int(split),
                                         int(width), int(height), _p(F_out), _p(B_out),
                                         int(out_dtype)))


def abcd_render_refresh_packed(ctx: Context, cam, opts, proj, tiles, tile_map, packed, count):
    """K10 into a packed layer: tile_map int32 [tiles], packed fp16 [tiles][16][16][4],
    count int32 [1] (CUDA tensors)."""
    p = proj.c(); t = tiles.c()
    ctx.check(lib().abcd_render_refresh_packed(ctx.h, C.byref(cam), _opt(opts), C.byref(p),
                                               C.byref(t), _p(tile_map), _p(packed), _p(count)))


def abcd_composite_cache_packed(ctx: Context, tile_maps, packed, order, split, width, height,
                                F_out, B_out, out_dtype=ABCD_F16):
    """tile_maps / packed: lists of CUDA tensors (None at the active position)."""
    L = len(tile_maps)
    maps = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in tile_maps])
    data = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in packed])
    ordr = (C.c_int * max(1, L))(*[int(k) for k in order])
    ctx.check(lib().abcd_composite_cache_packed(ctx.h, maps, data, L, ordr, int(split), int(width),
                                                int(height), _p(F_out), _p(B_out), int(out_dtype)))


def abcd_composite_fold_packed(ctx: Context, tile_maps, packed, width, height, acc_in=None,
                               acc_out=None, out16=None):
    """One side of K1 in pieces: acc_out = acc_in over the given packed layers, in list order
    (CUDA tensors; acc fp32 [H][W][4], out16 fp16 [H][W][4])."""
    n = len(tile_maps)
    maps = (C.c_void_p * max(1, n))(*[t.data_ptr() for t in tile_maps])
    data = (C.c_void_p * max(1, n))(*[t.data_ptr() for t in packed])
    ctx.check(lib().abcd_composite_fold_packed(ctx.h, maps, data, n, int(width), int(height),
                                               _p(acc_in), _p(acc_out), _p(out16)))


def abcd_layer_visibility(ctx: Context, layers, order, width, height, visible, coverage=None):
    """layers: list of L fp16 CUDA tensors [H][W][4] (None for a layer not in `order`); order:
    the layers front to back; visible / coverage: float64 CUDA tensors [L]."""
    L = len(layers)
    arr = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in layers])
    ordr = (C.c_int * max(1, len(order)))(*[int(k) for k in order])
    ctx.check(lib().abcd_layer_visibility(ctx.h, arr, L, ordr, len(order), int(width), int(height),
                                          _p(visible), _p(coverage)))


def abcd_layer_visibility_packed(ctx: Context, tile_maps, packed, order, width, height, visible,
                                 coverage=None):
    """The same over packed layers (tile_maps / packed: lists of CUDA tensors)."""
    L = len(tile_maps)
    maps = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in tile_maps])
    data = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in packed])
    ordr = (C.c_int * max(1, len(order)))(*[int(k) for k in order])
    ctx.check(lib().abcd_layer_visibility_packed(ctx.h, maps, data, L, ordr, len(order), int(width),
                                                 int(height), _p(visible), _p(coverage)))


def abcd_layer_visibility_tables(ctx: Context, pl, width, height, visible, coverage=None):
    """abcd_layer_visibility_packed over the tables of a PackedLayers built with split = L
    (every layer of the order, front to back)."""
    ctx.check(lib().abcd_layer_visibility_packed(ctx.h, pl.maps, pl.data, pl.L, pl.order, pl.L,
                                                 int(width), int(height), _p(visible),
                                                 _p(coverage)))


def cull_pairs(visible, coverage, tau_visible, tau_area=0.0):
    """Camera-partition pairs to keep (Section 4's visibility threshold and occlusion culling):
    a layer stays when its visible share of the composite is at least tau_visible and its
    image area at least tau_area.  The dropped layers' visible shares add up to a bound on the
    mean per-channel error of the culled composite.  Host arrays in, boolean mask out."""
    import numpy as np
    v, c = np.asarray(visible, dtype=np.float64), np.asarray(coverage, dtype=np.float64)
    return (v >= float(tau_visible)) & (c >= float(tau_area))


class TrainStep:
    """abcd_train_step with the argument structs built once: the buffers of a training loop
    stay put, so only the camera, F, B, target, loss slot and step change per call."""

    def __init__(self, ctx: Context, theta, grads, m, v, proj, tiles, out_rgba, state, lr,
                 beta1=0.9, beta2=0.999, eps=1e-15, lambda_ssim=0.2, opts=None, bg=None):
        self.ctx = ctx
        self.structs = [theta.c(), grads.c(), m.c(), v.c(), proj.c(), tiles.c(), state.c()]
        self.refs = [C.byref(x) for x in self.structs]
        self.opts = _opt(opts)
        self.bg = _bg(bg)
        self.out = _p(out_rgba)
        self.lr = (C.c_float * 6)(*[float(x) for x in lr])
        self.beta1, self.beta2, self.eps, self.lam = float(beta1), float(beta2), float(eps), float(lambda_ssim)
        self.keep = (theta, grads, m, v, proj, tiles, out_rgba, state)

    def __call__(self, cam, F, B, gt_rgb, loss_out, step, fb_dtype=ABCD_F16):
        th, gr, mm, vv, pr, ti, st = self.refs
        self.ctx.check(lib().abcd_train_step(
            self.ctx.h, th, gr, mm, vv, C.byref(cam), self.opts, pr, ti, _p(F), _p(B), int(fb_dtype),
            self.bg, self.out, st, _p(gt_rgb), self.lam, _p(loss_out), self.lr, self.beta1,
            self.beta2, self.eps, int(step)))


class RefreshLayer:
    """abcd_refresh_layer with the argument structs of one context's buffers built once."""

    def __init__(self, ctx: Context, theta, proj, tiles, opts=None):
        self.ctx = ctx
        self.structs = [theta.c(), proj.c(), tiles.c()]
        self.refs = [C.byref(x) for x in self.structs]
        self.opts = _opt(opts)
        self.keep = (theta, proj, tiles)

    def __call__(self, cam, tile_map, packed, count):
        th, pr, ti = self.refs
        self.ctx.check(lib().abcd_refresh_layer(self.ctx.h, th, C.byref(cam), self.opts, pr, ti,
                                                _p(tile_map), _p(packed), _p(count)))


class PackedLayers:
    """The pointer tables of one camera's packed layers, built once for repeated composites
    (the per-call conversion of 2 L tensors is host time a stage spends per camera)."""

    def __init__(self, tile_maps, packed, order, split):
        L = len(tile_maps)
        self.L, self.split = L, int(split)
        self.maps = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in tile_maps])
        self.data = (C.c_void_p * max(1, L))(*[(t.data_ptr() if t is not None else None) for t in packed])
        self.order = (C.c_int * max(1, L))(*[int(k) for k in order])
        self.keep = (tile_maps, packed)          # the tensors must outlive the tables


def abcd_composite_cache_packed_tables(ctx: Context, pl: PackedLayers, width, height, F_out, B_out,
                                       out_dtype=ABCD_F16):
    ctx.check(lib().abcd_composite_cache_packed(ctx.h, pl.maps, pl.data, pl.L, pl.order, pl.split,
                                                int(width), int(height), _p(F_out), _p(B_out),
                                                int(out_dtype)))


def abcd_cache_fetch(ctx: Context, slot, host_src, dev_dst, nbytes=None):
    """Queue host_src (pinned host tensor) -> dev_dst (CUDA tensor) for `slot`."""
    n = host_src.numel() * host_src.element_size() if nbytes is None else int(nbytes)
    ctx.check(lib().abcd_cache_fetch(ctx.h, int(slot), _hp(host_src), _p(dev_dst), n))


def abcd_cache_wait(ctx: Context, slot):
    ctx.check(lib().abcd_cache_wait(ctx.h, int(slot)))


def abcd_cache_release(ctx: Context, slot):
    ctx.check(lib().abcd_cache_release(ctx.h, int(slot)))


def abcd_cache_store(ctx: Context, slot, dev_src, host_dst, nbytes=None):
    """Queue dev_src (CUDA tensor) -> host_dst (pinned host tensor) for `slot`, after the
    stream's work."""
    n = dev_src.numel() * dev_src.element_size() if nbytes is None else int(nbytes)
    ctx.check(lib().abcd_cache_store(ctx.h, int(slot), _p(dev_src), _hp(host_dst), n))


def abcd_cache_sync(ctx: Context):
    ctx.check(lib().abcd_cache_sync(ctx.h))


def abcd_assign_cells(means_np, origin, side, dims):
    import numpy as np
    m = np.ascontiguousarray(means_np, dtype=np.float32)
    n = m.shape[0]
    cell = np.zeros(n, np.int32)
    o = (C.c_double * 3)(*[float(v) for v in origin])
    d = (C.c_int * 3)(*[int(v) for v in dims])
    st = lib().abcd_assign_cells(m.ctypes.data_as(C.c_void_p), n, o, float(side), d,
                                 cell.ctypes.data_as(C.c_void_p))
    if st != ABCD_OK:
        raise AbcdError(st, "abcd_assign_cells")
    return cell


def abcd_partition_split(dims, origin, side, campos, active):
    import numpy as np
    total = int(np.prod(dims))
    front, back = np.zeros(total, np.int32), np.zeros(total, np.int32)
    nf, nb = C.c_int(), C.c_int()
    st = lib().abcd_partition_split((C.c_int * 3)(*[int(v) for v in dims]),
                                    (C.c_double * 3)(*[float(v) for v in origin]), float(side),
                                    (C.c_double * 3)(*[float(v) for v in campos]), int(active),
                                    front.ctypes.data_as(C.c_void_p), C.byref(nf),
                                    back.ctypes.data_as(C.c_void_p), C.byref(nb))
    if st != ABCD_OK:
        raise AbcdError(st, "abcd_partition_split")
    return front[:nf.value].copy(), back[:nb.value].copy()


def abcd_measure_alu_peaks(device=0) -> dict:
    """Measured fp32 FMA (scalar and packed) and ex2.approx throughput of `device` (a few short
    timed kernels; no clock or device setting is changed)."""
    p = abcd_alu_peaks()
    st = lib().abcd_measure_alu_peaks(int(device), C.byref(p))
    if st != ABCD_OK:
        raise AbcdError(st, "abcd_measure_alu_peaks")
    return {k: getattr(p, k) for k, _ in abcd_alu_peaks._fields_}


def abcd_block_bounds(ctx: Context, theta: Gaussians, box):
    """box: CUDA float tensor [6] (lowest x, y, z, highest x, y, z of the 3-sigma ellipsoids)."""
    g = theta.c()
    ctx.check(lib().abcd_block_bounds(ctx.h, C.byref(g), _p(box)))


def abcd_pair_visible(cam: abcd_camera, box, opts=None) -> bool:
    """Whether the partition with extent `box` (6 floats: lowest, highest corner) may be seen."""
    b = (C.c_double * 6)(*[float(v) for v in box])
    v = C.c_int()
    st = lib().abcd_pair_visible(C.byref(cam), _opt(opts), b, C.byref(v))
    if st != ABCD_OK:
        raise AbcdError(st, "abcd_pair_visible")
    return bool(v.value)


def visible_pairs(ctx: Context, blocks, cameras, dims, origin, side, opts=None):
    """Visibility of every (camera, block) pair: [C][n_blocks] bool; a block's extent is its
    cell united with its Gaussians' 3-sigma box (blocks: {block id: Gaussians on the device};
    absent or empty blocks are not visible)."""
    import numpy as np
    torch = _torch()
    n_blocks = int(np.prod(dims))
    out = np.zeros((len(cameras), n_blocks), bool)
    boxes = {}
    for b, th in blocks.items():
        if th.n == 0:
            continue
        dev = torch.empty(6, device="cuda")
        abcd_block_bounds(ctx, th, dev)
        boxes[b] = dev
    ctx.sync()
    gx, gy = int(dims[0]), int(dims[1])
    cams = [c if isinstance(c, abcd_camera) else camera(c) for c in cameras]
    for b, dev in boxes.items():
        bx = dev.cpu().numpy().astype(np.float64)
        ijk = np.array([b % gx, (b // gx) % gy, b // (gx * gy)], np.float64)
        lo = np.asarray(origin, np.float64) + side * ijk
        box = np.concatenate([np.minimum(bx[:3], lo), np.maximum(bx[3:], lo + side)])
        for ci, cam in enumerate(cams):
            out[ci, b] = abcd_pair_visible(cam, box, opts)
    return out
