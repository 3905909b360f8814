"""Seeded synthetic inputs shaped like the paper's workloads (Section 3: about 200 training
cameras around a scene cut by a regular grid of side 5 units).

This module only draws inputs: Gaussian parameters, pinhole cameras, target images and
cached-layer stand-ins.  It holds none of the method's arithmetic (no projection, no
blending, no partition assignment, no loss); both the CUDA path and the CPU oracle consume
its arrays unchanged.  Every array it returns is float32 (or an integer type), so the fp64
oracle sees exactly the values the kernels see.

Distributions (the workload recipe):
  * means: uniform inside each grid cell (a block of ``per_cell`` Gaussians per cell), or, for
    the stress workload, a 16-component isotropic Gaussian mixture;
  * log-scales: N(log(0.05 * side), 0.5) per axis;
  * rotations: normalised N(0, I4) quaternions, (w, x, y, z) order;
  * opacity logits: N(0, 1)  (so opacity = sigmoid(N(0, 1)));
  * colour: the degree-0 coefficient uniform on [-sqrt(pi), sqrt(pi)], the range whose
    view-independent colour term lies in [0, 1]; higher-degree coefficients N(0, 0.05);
  * cameras: pinhole, 60 degree horizontal field of view, principal point at the image
    centre, world z up, looking at the scene centre from a ring (optionally with height
    jitter) or from Fibonacci points on the upper hemisphere, at 1.5x the scene half-diagonal.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np


@dataclass
class Camera:
    """World-to-camera rigid transform (x right, y down, z forward) and pinhole intrinsics."""
    R: np.ndarray          # (3, 3) float32, row-major
    t: np.ndarray          # (3,) float32
    fx: float
    fy: float
    cx: float
    cy: float
    width: int
    height: int

    @property
    def position(self) -> np.ndarray:
        """Camera centre in world coordinates (float64)."""
        R = self.R.astype(np.float64)
        return -R.T @ self.t.astype(np.float64)


@dataclass
class Gaussians:
    means: np.ndarray           # (N, 3) float32
    log_scales: np.ndarray      # (N, 3) float32
    quats: np.ndarray           # (N, 4) float32, (w, x, y, z), not necessarily unit
    opacity_logits: np.ndarray  # (N,)  float32
    sh: np.ndarray              # (N, D, 3) float32, D = (sh_degree + 1) ** 2
    sh_degree: int

    @property
    def n(self) -> int:
        return int(self.means.shape[0])

    def subset(self, idx) -> "Gaussians":
        return Gaussians(self.means[idx].copy(), self.log_scales[idx].copy(),
                         self.quats[idx].copy(), self.opacity_logits[idx].copy(),
                         self.sh[idx].copy(), self.sh_degree)

    def arrays(self):
        return (self.means, self.log_scales, self.quats, self.opacity_logits, self.sh)


@dataclass
class Grid:
    dims: tuple                 # (gx, gy, gz) cells
    side: float                 # cell edge length
    origin: np.ndarray          # (3,) float64, minimum corner

    @property
    def n_cells(self) -> int:
        return int(np.prod(self.dims))

    def cell_bounds(self, linear_id: int):
        gx, gy, _ = self.dims
        i = linear_id % gx
        j = (linear_id // gx) % gy
        k = linear_id // (gx * gy)
        lo = self.origin + self.side * np.array([i, j, k], dtype=np.float64)
        return lo, lo + self.side


@dataclass
class Scene:
    grid: Grid
    gaussians: Gaussians
    cameras: list = field(default_factory=list)
    block_of: np.ndarray = None   # (N,) cell the generator drew each Gaussian in


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(seed), int(stream)]))


def look_at(position, target, width, height, fov_x_deg=60.0, up=(0.0, 0.0, 1.0)) -> Camera:
    """Pinhole camera at ``position`` looking at ``target`` (x right, y down, z forward)."""
    p = np.asarray(position, dtype=np.float64)
    f = np.asarray(target, dtype=np.float64) - p
    f /= np.linalg.norm(f)
    r = np.cross(f, np.asarray(up, dtype=np.float64))
    if np.linalg.norm(r) < 1e-9:          # looking straight up/down: pick any right vector
        r = np.cross(f, np.array([1.0, 0.0, 0.0]))
    r /= np.linalg.norm(r)
    d = np.cross(f, r)
    R = np.stack([r, d, f]).astype(np.float32)
    t = (-R.astype(np.float64) @ p).astype(np.float32)
    fx = np.float32(0.5 * width / math.tan(math.radians(fov_x_deg) / 2.0))
    return Camera(R=R, t=t, fx=float(fx), fy=float(fx), cx=float(np.float32(width / 2.0)),
                  cy=float(np.float32(height / 2.0)), width=int(width), height=int(height))


def ring_cameras(n, radius, center, width, height, seed, height_jitter=0.0, fov=60.0):
    rng = _rng(seed, 7)
    cams = []
    for i in range(n):
        a = 2.0 * math.pi * i / n
        z = center[2] + (rng.uniform(-height_jitter, height_jitter) if height_jitter > 0 else 0.0)
        pos = np.array([center[0] + radius * math.cos(a), center[1] + radius * math.sin(a), z])
        cams.append(look_at(pos, center, width, height, fov))
    return cams


def inside_cameras(grid, n, width, height, seed, fov=60.0):
    """n cameras inside the grid's box (walk-through views): positions uniform in the middle
    80% of the box, looking horizontally in a uniform direction."""
    rng = _rng(seed, 7)
    lo = np.asarray(grid.origin, np.float64)
    hi = lo + grid.side * np.asarray(grid.dims, np.float64)
    cams = []
    for _ in range(n):
        p = lo + (0.1 + 0.8 * rng.random(3)) * (hi - lo)
        yaw = rng.uniform(0.0, 2.0 * np.pi)
        cams.append(look_at(p, p + np.array([np.cos(yaw), np.sin(yaw), 0.0]), width, height,
                            fov_x_deg=fov))
    return cams


def hemisphere_cameras(n, radius, center, width, height, fov=60.0):
    cams = []
    golden = math.pi * (3.0 - math.sqrt(5.0))
    for i in range(n):
        z = 0.05 + 0.9 * (i + 0.5) / n          # upper hemisphere, away from the pole
        rr = math.sqrt(max(0.0, 1.0 - z * z))
        a = golden * i
        pos = np.asarray(center) + radius * np.array([rr * math.cos(a), rr * math.sin(a), z])
        cams.append(look_at(pos, center, width, height, fov))
    return cams


def _gaussian_params(rng, n, side, sh_degree, means):
    D = (sh_degree + 1) ** 2
    log_scales = rng.normal(math.log(0.05 * side), 0.5, size=(n, 3)).astype(np.float32)
    q = rng.normal(size=(n, 4))
    q /= np.linalg.norm(q, axis=1, keepdims=True)
    logits = rng.normal(0.0, 1.0, size=n).astype(np.float32)
    sh = np.zeros((n, D, 3), dtype=np.float32)
    sh[:, 0, :] = rng.uniform(-math.sqrt(math.pi), math.sqrt(math.pi), size=(n, 3))
    if D > 1:
        sh[:, 1:, :] = rng.normal(0.0, 0.05, size=(n, D - 1, 3))
    return Gaussians(means.astype(np.float32), log_scales, q.astype(np.float32), logits, sh,
                     sh_degree)


def grid_scene(dims, side, per_cell, sh_degree, seed) -> Scene:
    """Gaussians drawn uniformly inside each cell of a regular grid centred on the origin."""
    dims = tuple(int(d) for d in dims)
    origin = -0.5 * side * np.asarray(dims, dtype=np.float64)
    grid = Grid(dims, float(side), origin)
    rng = _rng(seed, 1)
    n_cells = grid.n_cells
    means = np.empty((n_cells * per_cell, 3), dtype=np.float64)
    block_of = np.repeat(np.arange(n_cells, dtype=np.int32), per_cell)
    for c in range(n_cells):
        lo, hi = grid.cell_bounds(c)
        means[c * per_cell:(c + 1) * per_cell] = rng.uniform(lo, hi, size=(per_cell, 3))
    # keep every mean strictly inside its cell after rounding to float32
    m32 = means.astype(np.float32)
    for c in range(n_cells):
        lo, hi = grid.cell_bounds(c)
        sl = slice(c * per_cell, (c + 1) * per_cell)
        eps = 1e-4 * side
        m32[sl] = np.clip(m32[sl], (lo + eps).astype(np.float32), (hi - eps).astype(np.float32))
    g = _gaussian_params(rng, n_cells * per_cell, side, sh_degree, m32)
    return Scene(grid=grid, gaussians=g, block_of=block_of)


def mixture_block(n, extent, n_blobs, sh_degree, seed, side=5.0) -> Gaussians:
    """One dense block: means from an isotropic Gaussian mixture (stress workload)."""
    rng = _rng(seed, 2)
    centres = rng.uniform(-0.5 * extent, 0.5 * extent, size=(n_blobs, 3))
    comp = rng.integers(0, n_blobs, size=n)
    means = centres[comp] + rng.normal(0.0, 0.05 * extent, size=(n, 3))
    return _gaussian_params(rng, n, side, sh_degree, means.astype(np.float32))


def perturbed(g: Gaussians, side: float, seed: int) -> Gaussians:
    """Seed-perturbed copy used to render target images."""
    rng = _rng(seed, 3)
    out = g.subset(slice(None))
    out.means = (g.means + rng.normal(0.0, 0.02 * side, size=g.means.shape)).astype(np.float32)
    out.sh = g.sh.copy()
    out.sh[:, 0, :] += rng.normal(0.0, 0.05 * 2.0 * math.sqrt(math.pi),
                                  size=(g.n, 3)).astype(np.float32)
    out.opacity_logits = (g.opacity_logits +
                          rng.normal(0.0, 0.2, size=g.n)).astype(np.float32)
    return out


def premultiplied_layers(n_layers, height, width, seed):
    """Random premultiplied RGBA layers: a ~ U[0, 1], rgb = a * U[0, 1]^3 (float32)."""
    rng = _rng(seed, 4)
    a = rng.uniform(0.0, 1.0, size=(n_layers, height, width, 1))
    rgb = a * rng.uniform(0.0, 1.0, size=(n_layers, height, width, 3))
    return np.concatenate([rgb, a], axis=-1).astype(np.float32)


def random_image(height, width, channels, seed, lo=0.0, hi=1.0):
    rng = _rng(seed, 5)
    return rng.uniform(lo, hi, size=(height, width, channels)).astype(np.float32)


def random_permutation(n, seed):
    return _rng(seed, 6).permutation(n).astype(np.int32)


# --------------------------------------------------------------------------------------
# Named workloads (sizes from the paper-shaped configurations).

def half_diagonal(grid: Grid) -> float:
    return 0.5 * grid.side * float(np.linalg.norm(np.asarray(grid.dims, dtype=np.float64)))


def tiny_scene(seed=1001, per_cell=2000, res=128, n_cams=4) -> Scene:
    """2x2x2 grid x 2,000 Gaussians per cell, SH degree 0, 4 ring cameras at 128x128."""
    s = grid_scene((2, 2, 2), 5.0, per_cell, 0, seed)
    s.cameras = ring_cameras(n_cams, 1.5 * half_diagonal(s.grid), np.zeros(3), res, res, seed)
    return s


def medium_scene(seed=1002, per_cell=20000, width=640, height=480, n_cams=50) -> Scene:
    """3x3x3 grid x 20,000 Gaussians per cell, SH degree 3, 50 hemisphere cameras 640x480."""
    s = grid_scene((3, 3, 3), 5.0, per_cell, 3, seed)
    s.cameras = hemisphere_cameras(n_cams, 1.5 * half_diagonal(s.grid), np.zeros(3),
                                   width, height)
    return s


def scene_scale(seed=1003, per_cell=100000, width=1237, height=822, n_cams=200) -> Scene:
    """4x4x2 grid x 100,000 Gaussians per cell (3.2M), SH degree 3, 200 ring cameras at
    1237x822 with height jitter of +-10% of the vertical extent."""
    s = grid_scene((4, 4, 2), 5.0, per_cell, 3, seed)
    ez = s.grid.dims[2] * s.grid.side
    s.cameras = ring_cameras(n_cams, 1.5 * half_diagonal(s.grid), np.zeros(3), width, height,
                             seed, height_jitter=0.1 * ez)
    return s
