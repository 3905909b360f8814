"""Block coordinate descent over every partition of the grid (Section 2), in cyclic order.

A stage trains one block for T steps: the cached renders of the frozen blocks, taken in each
camera's depth order, are composited into F and B (abcd_composite_cache), each step renders
the active block alone and composites F over A over B (abcd_train_step), and at the end the
block's cached renders are refreshed (abcd_render_composite_fwd's refresh output).  Two
variants share the schedule: "ablated" trains each block with F = B = transparent, as if it
were the whole scene (the ablation of Section 3), and a one-block grid is plain full-scene
training, the reference both are compared with.  Host orchestration of the C ABI only:
every operation runs in libabcd's kernels.
"""
from __future__ import annotations

import numpy as np

from . import (ABCD_F16, ABCD_F32, Context, FwdState, Gaussians, Projected, Tiles, TrainStep,
               abcd_assign_cells, abcd_composite_cache, abcd_layer_visibility, abcd_loss,
               abcd_partition_split, abcd_project, abcd_bin_sort, abcd_render_composite_fwd,
               camera, cull_pairs, _torch)

# Adam learning rates per group (means, log-scales, quaternions, opacity logits, SH degree 0,
# higher SH degrees): 3DGS-style defaults, the means' scaled by the scene extent.
def default_lr(extent):
    return [1.6e-4 * extent, 5e-3, 1e-3, 0.025, 2.5e-3, 2.5e-3 / 20]


class BCD:
    """Cyclic block coordinate descent over the cells of a regular grid.

    gaussians: scenegen.Gaussians of the whole scene; dims, origin, side: the grid; cameras:
    objects with R, t, fx, fy, cx, cy, width, height, position; targets: float32 [C][H][W][3];
    mode: "abcd" (F and B from the cache) or "ablated" (F = B = transparent).  cull_tau: the
    visibility threshold of Section 5's culling of camera-partition pairs (None: no culling):
    after every refresh each camera's layers are measured (abcd_layer_visibility) and a pair
    whose visible share of the camera's composite is below cull_tau is dropped, from F and B
    of the other blocks' stages and from the cameras its own block trains on, until a later
    measurement brings it back."""

    def __init__(self, gaussians, dims, origin, side, cameras, targets, T, lr, mode="abcd",
                 device=0, seed=0, lambda_ssim=0.2, max_pairs=2_000_000, cull_tau=None):
        assert mode in ("abcd", "ablated")
        torch = _torch()
        self.torch, self.mode, self.T = torch, mode, int(T)
        self.lam = float(lambda_ssim)
        self.ctx = Context(device)
        self.dims = tuple(int(d) for d in dims)
        self.origin = [float(v) for v in origin]
        self.side = float(side)
        n_blocks = int(np.prod(self.dims))
        cells = abcd_assign_cells(gaussians.means, self.origin, self.side, self.dims)
        self.members = [np.nonzero(cells == b)[0] for b in range(n_blocks)]
        self.blocks = [b for b in range(n_blocks) if len(self.members[b])]
        self.theta = {b: Gaussians.from_numpy(gaussians.subset(self.members[b])) for b in self.blocks}
        n_max = max(len(self.members[b]) for b in self.blocks)
        self.cams_np = list(cameras)
        self.cams = [camera(c) for c in cameras]
        W, H = int(cameras[0].width), int(cameras[0].height)
        self.W, self.H = W, H
        self.ctx.reserve(n_max, max_pairs, W * H)
        self.proj = Projected.alloc(n_max)
        self.tiles = Tiles.alloc(max_pairs, W, H)
        self.out = torch.empty(H, W, 4, device="cuda")
        self.state = FwdState.alloc(W, H)
        C = len(cameras)
        self.gt = torch.from_numpy(np.ascontiguousarray(targets, dtype=np.float32)).cuda()
        self.layers = torch.zeros(C, n_blocks, H, W, 4, dtype=torch.float16, device="cuda")
        self.F = torch.zeros(C, H, W, 4, dtype=torch.float16, device="cuda")
        self.B = torch.zeros_like(self.F)
        self.order = {}                      # (camera, block) -> (front-to-back order, split)
        for ci, c in enumerate(cameras):
            for b in range(n_blocks):
                f, bk = abcd_partition_split(self.dims, self.origin, self.side, c.position, b)
                self.order[ci, b] = (list(f) + [b] + list(bk), len(f))
        self.lr = list(lr)
        self.rng = np.random.default_rng(seed)
        self.queue = []
        self.loss = torch.zeros(max(1, self.T), device="cuda")
        self.steps_done = 0
        self.cull_tau = cull_tau
        self.keep = np.ones((C, n_blocks), bool)     # camera-partition pairs in use
        self.visible = np.zeros((C, n_blocks))
        for b in self.blocks:
            self.refresh(b, measure=False)
        self.measure_visibility()

    # ---- pieces of a stage
    def refresh(self, b, measure=True):
        """Re-renders block b's cached layer for every camera (K2-K5, refresh output), then
        (with culling) measures the cameras' layers again."""
        th = self.theta[b]
        for ci, cam in enumerate(self.cams):
            abcd_project(self.ctx, th, cam, None, self.proj)
            abcd_bin_sort(self.ctx, self.proj, th.n, cam, self.tiles)
            abcd_render_composite_fwd(self.ctx, cam, None, self.proj, self.tiles,
                                      refresh_f16=self.layers[ci, b])
        if measure:
            self.measure_visibility()

    def measure_visibility(self):
        """Visible share of every camera-partition pair in its camera's composite of all
        cached layers, and the pairs kept at the threshold."""
        if self.cull_tau is None:
            return
        torch = self.torch
        C, n_blocks = self.keep.shape
        vis = torch.empty(C, n_blocks, dtype=torch.float64, device="cuda")
        cov = torch.empty_like(vis)
        for ci in range(C):
            order, _ = self.order[ci, 0]
            abcd_layer_visibility(self.ctx, [self.layers[ci, k] for k in range(n_blocks)], order,
                                  self.W, self.H, vis[ci], cov[ci])
        self.visible = vis.cpu().numpy()
        self.keep = cull_pairs(self.visible, cov.cpu().numpy(), self.cull_tau)

    def composite(self, b):
        """F and B of every camera around active block b, from the cached layers of the pairs
        in use (K1)."""
        for ci in range(len(self.cams)):
            order, _ = self.order[ci, b]
            kept = [k for k in order if k == b or self.keep[ci, k]]
            split = kept.index(b)
            lay = [self.layers[ci, k] if k != b else None for k in kept]
            abcd_composite_cache(self.ctx, lay, list(range(len(kept))), split, self.W, self.H,
                                 self.F[ci], self.B[ci])

    def cameras_of(self, b):
        """Cameras block b trains on: those whose pair with b is in use."""
        return [ci for ci in range(len(self.cams)) if self.keep[ci, b]]

    def next_camera(self, allowed=None):
        """Shuffle without replacement over the allowed cameras, reshuffled when used up."""
        allowed = list(range(len(self.cams))) if allowed is None else list(allowed)
        self.queue = [ci for ci in self.queue if ci in allowed]
        if not self.queue:
            self.queue = [allowed[i] for i in self.rng.permutation(len(allowed))]
        return int(self.queue.pop())

    def stage(self, b):
        th = self.theta[b]
        torch = self.torch
        grads, m, v = (Gaussians.zeros_like(th) for _ in range(3))   # Adam state per stage
        if self.mode == "abcd":
            self.composite(b)
        step = TrainStep(self.ctx, th, grads, m, v, self.proj, self.tiles, self.out, self.state,
                         self.lr, lambda_ssim=self.lam)
        allowed = self.cameras_of(b)
        for t in range(self.T if allowed else 0):
            ci = self.next_camera(allowed)
            F = self.F[ci] if self.mode == "abcd" else None
            B = self.B[ci] if self.mode == "abcd" else None
            step(self.cams[ci], F, B, self.gt[ci], self.loss[t:t + 1], t + 1)
        self.steps_done += self.T if allowed else 0
        self.refresh(b)

    def cycle(self):
        for b in self.blocks:
            self.stage(b)

    # ---- evaluation
    def render_full(self, ci):
        """The full render of camera ci: every block's cached layer composited in the camera's
        depth order (fp32 RGBA)."""
        torch = self.torch
        n_blocks = self.layers.shape[1]
        order, _ = self.order[ci, 0]
        full = torch.empty(self.H, self.W, 4, device="cuda")
        abcd_composite_cache(self.ctx, [self.layers[ci, k] for k in range(n_blocks)], order,
                             n_blocks, self.W, self.H, full, None, ABCD_F16, ABCD_F32)
        return full

    def eval_loss(self):
        """Mean over cameras of the loss of the full render against the target."""
        torch = self.torch
        acc = torch.zeros(len(self.cams), device="cuda")
        for ci in range(len(self.cams)):
            full = self.render_full(ci)
            abcd_loss(self.ctx, full, self.gt[ci], self.W, self.H, self.lam, acc[ci:ci + 1], None)
        self.ctx.sync()
        return float(acc.mean().item())


def quality_experiment(T=100, cycles=3, per_cell=1000, n_cams=8, width=96, height=72, seed=2024,
                       cull_tau=0.01):
    """Section 3's comparison on a seeded synthetic scene (a 2x2x1 grid of side 5, SH degree
    0): full-scene training (one block, 4 T steps per cycle), ABCD and the ablated variant (4
    blocks, T steps each per cycle), the same number of steps in all three, against targets
    rendered from a perturbed copy of the scene; and ABCD with the camera-partition pairs
    culled at visible share cull_tau (Section 5), which trains each block on the cameras that
    see it.  Returns {name: [eval loss after 0..cycles]}; the eval renders every layer."""
    from . import scenegen as sg
    dims, side = (2, 2, 1), 5.0
    s = sg.grid_scene(dims, side, per_cell, 0, seed=seed)
    s.cameras = sg.ring_cameras(n_cams, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), width, height,
                                seed=seed, height_jitter=1.0)
    origin = s.grid.origin
    blank = np.zeros((n_cams, height, width, 3), np.float32)
    ref = BCD(sg.perturbed(s.gaussians, side, seed=seed + 1), (1, 1, 1), origin, 2 * side,
              s.cameras, blank, 0, default_lr(2 * side))
    targets = np.stack([ref.render_full(ci)[..., :3].cpu().numpy() for ci in range(n_cams)])
    out = {}
    for name, d, sd, mode, t, tau in (("full_scene", (1, 1, 1), 2 * side, "abcd", 4 * T, None),
                                      ("abcd", dims, side, "abcd", T, None),
                                      ("ablated", dims, side, "ablated", T, None),
                                      ("abcd_culled", dims, side, "abcd", T, cull_tau)):
        run = BCD(s.gaussians, d, origin, sd, s.cameras, targets, t, default_lr(2 * side),
                  mode=mode, seed=seed + 2, cull_tau=tau)
        hist = [run.eval_loss()]
        for _ in range(cycles):
            run.cycle()
            hist.append(run.eval_loss())
        out[name] = hist
    return out
