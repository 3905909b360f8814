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
               abcd_adam_active, abcd_assign_cells, abcd_backward, abcd_composite_cache,
               abcd_layer_visibility, abcd_loss, abcd_partition_split, abcd_project,
               abcd_bin_sort, abcd_render_composite_fwd, camera, cull_pairs, visible_pairs,
               _torch)

# Adam learning rates per group (means, log-scales, quaternions, opacity logits, SH degree 0,
# higher SH degrees): 3DGS-style defaults, the means' scaled by the scene extent.
def default_lr(extent):
    return [1.6e-4 * extent, 5e-3, 1e-3, 0.025, 2.5e-3, 2.5e-3 / 20]


def halo_members(means, members, blocks, b, dims, origin, side, margin):
    """The halo of block b: {other block q: positions, in q's member list, of q's Gaussians
    whose means lie within `margin` of b's cell (the closed box widened by margin on every
    side)}.  Cells are numbered x + dims[0] (y + dims[1] z)."""
    gx, gy, _ = dims
    ix, iy, iz = b % gx, (b // gx) % gy, b // (gx * gy)
    lo = np.asarray(origin, np.float64) + side * np.array([ix, iy, iz], np.float64)
    hi = lo + side
    out = {}
    for q in blocks:
        if q == b:
            continue
        mq = np.asarray(means, np.float64)[members[q]]
        near = np.all((mq >= lo - margin) & (mq <= hi + margin), axis=1)
        if near.any():
            out[q] = np.nonzero(near)[0]
    return out


class BCD:
    """Cyclic block coordinate descent over the cells of a regular grid.

    gaussians: scenegen.Gaussians of the whole scene; dims, origin, side: the grid; cameras:
    objects with R, t, fx, fy, cx, cy, width, height, position; targets: float32 [C][H][W][3];
    mode: "abcd" (F and B from the cache) or "ablated" (F = B = transparent).  cull_tau: the
    visibility threshold of Section 4's culling of camera-partition pairs (None: no culling):
    after every refresh each camera's layers are measured (abcd_layer_visibility) and a pair
    whose visible share of the camera's composite is below cull_tau is dropped, from F and B
    of the other blocks' stages and from the cameras its own block trains on, until a later
    measurement brings it back.  overlap: the width of the overlapping boundary region that
    Section 4 proposes (0: none).  Membership stays by the mean, but a block's stage renders,
    with the block, the other blocks' Gaussians whose means lie within `overlap` of its cell
    (its halo: frozen, sorted by depth together with the block's own, no gradient step), and
    for every camera F and B take each donor block's layer re-rendered without them, so every
    Gaussian is drawn once and the ones near the block's faces in their true depth order."""

    def __init__(self, gaussians, dims, origin, side, cameras, targets, T, lr, mode="abcd",
                 device=0, seed=0, lambda_ssim=0.2, max_pairs=2_000_000, cull_tau=None,
                 overlap=0.0):
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
        # halo of each block: {donor block: positions in the donor's parameters}
        self.overlap = float(overlap)
        self.halo = {b: self._halo(b, np.asarray(gaussians.means, np.float64))
                     for b in self.blocks} if self.overlap > 0 else {b: {} for b in self.blocks}
        n_max = max(len(self.members[b]) + sum(len(v) for v in self.halo[b].values())
                    for b in self.blocks)
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
        self.frustum = np.ones((C, n_blocks), bool)  # pairs that pass the frustum filter
        self.update_frustum()
        for b in self.blocks:
            self.refresh(b, measure=False)
        self.measure_visibility()

    def _halo(self, b, means):
        return halo_members(means, self.members, self.blocks, b, self.dims, self.origin,
                            self.side, self.overlap)

    def _take(self, g, pos):
        """Gaussians at positions pos (host int array) of g, as new device tensors."""
        idx = self.torch.as_tensor(pos, dtype=self.torch.long, device="cuda")
        return Gaussians(*(t.index_select(0, idx) for t in g.tensors()), g.sh_degree)

    def _stage_theta(self, b):
        """Block b followed by its halo (one buffer), or block b itself without a halo."""
        th = self.theta[b]
        if not self.halo[b]:
            return th
        parts = [th] + [self._take(self.theta[q], pos) for q, pos in self.halo[b].items()]
        return Gaussians(*(self.torch.cat([p.tensors()[k] for p in parts]).contiguous()
                           for k in range(5)), th.sh_degree)

    def _core_layer(self, q, pos, ci, dst):
        """Donor block q's layer for camera ci without its Gaussians at positions pos."""
        keep = np.setdiff1d(np.arange(self.theta[q].n), pos)
        g = self._take(self.theta[q], keep)
        if g.n == 0:
            dst.zero_()
            return
        abcd_project(self.ctx, g, self.cams[ci], None, self.proj)
        abcd_bin_sort(self.ctx, self.proj, g.n, self.cams[ci], self.tiles)
        abcd_render_composite_fwd(self.ctx, self.cams[ci], None, self.proj, self.tiles,
                                  refresh_f16=dst)

    # ---- pieces of a stage
    def refresh(self, b, measure=True):
        """Re-renders block b's cached layer for every camera (K2-K5, refresh output), then
        (with culling) measures the cameras' layers again."""
        th = self.theta[b]
        for ci, cam in enumerate(self.cams):
            if not self.frustum[ci, b]:           # outside the frustum: transparent
                self.layers[ci, b].zero_()
                continue
            abcd_project(self.ctx, th, cam, None, self.proj)
            abcd_bin_sort(self.ctx, self.proj, th.n, cam, self.tiles)
            abcd_render_composite_fwd(self.ctx, cam, None, self.proj, self.tiles,
                                      refresh_f16=self.layers[ci, b])
        if measure:
            self.measure_visibility()

    def update_frustum(self):
        """a0: the camera-partition pairs whose partition (cell united with its Gaussians'
        3-sigma box) meets the camera's frustum; the others are never cached, composited or
        trained on (their layers are transparent)."""
        self.frustum = visible_pairs(self.ctx, self.theta, self.cams, self.dims, self.origin,
                                     self.side)
        if self.cull_tau is None:
            self.keep = self.frustum.copy()
        else:
            self.keep &= self.frustum

    def measure_visibility(self):
        """Visible share of every camera-partition pair in its camera's composite of all
        cached layers, and the pairs kept at the threshold (within the frustum's pairs)."""
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
        self.keep = cull_pairs(self.visible, cov.cpu().numpy(), self.cull_tau) & self.frustum

    def composite(self, b):
        """F and B of every camera around active block b, from the cached layers of the pairs
        in use (K1); with a halo, each donor block's layer is its layer without the halo."""
        core = self.torch.empty(len(self.halo[b]), self.H, self.W, 4, dtype=self.torch.float16,
                                device="cuda")
        for ci in range(len(self.cams)):
            order, _ = self.order[ci, b]
            kept = [k for k in order if k == b or self.keep[ci, k]]
            split = kept.index(b)
            lay = [self.layers[ci, k] if k != b else None for k in kept]
            for j, (q, pos) in enumerate(self.halo[b].items()):
                if q in kept:
                    self._core_layer(q, pos, ci, core[j])
                    lay[kept.index(q)] = core[j]
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

    def stage(self, b, trace=None):
        """One stage of block b: composite F and B (abcd mode), T steps, refresh.  trace, if
        given, is called after every step as trace(t, camera, theta, grads, m, v, loss) with the
        block's device tensors as they are after the step's Adam update (an observer: it must
        not change them)."""
        th = self.theta[b]
        grads, m, v = (Gaussians.zeros_like(th) for _ in range(3))   # Adam state per stage
        if self.mode == "abcd":
            self.composite(b)
        allowed = self.cameras_of(b)
        if self.halo[b]:
            # the block and its frozen halo are rendered together; Adam updates the block's
            # rows (the first th.n of every array) only
            ths = self._stage_theta(b)
            gs = Gaussians.zeros_like(ths)
            head = lambda g: Gaussians(*(t[:th.n] for t in g.tensors()), g.sh_degree)
            for t in range(self.T if allowed else 0):
                ci = self.next_camera(allowed)
                cam = self.cams[ci]
                F = self.F[ci] if self.mode == "abcd" else None
                B = self.B[ci] if self.mode == "abcd" else None
                abcd_project(self.ctx, ths, cam, None, self.proj)
                abcd_bin_sort(self.ctx, self.proj, ths.n, cam, self.tiles)
                abcd_render_composite_fwd(self.ctx, cam, None, self.proj, self.tiles, F, B,
                                          ABCD_F16, None, self.out, self.state)
                abcd_backward(self.ctx, ths, cam, None, self.proj, self.tiles, F, B, ABCD_F16,
                              None, self.out, self.state, self.gt[ci], self.lam,
                              self.loss[t:t + 1], None, gs)
                abcd_adam_active(self.ctx, head(ths), head(gs), m, v, self.lr, 0.9, 0.999,
                                 1e-15, t + 1)
                if trace is not None:
                    trace(t, ci, head(ths), head(gs), m, v, self.loss[t:t + 1])
            for a_, s_ in zip(th.tensors(), ths.tensors()):
                a_.copy_(s_[:th.n])
        else:
            step = TrainStep(self.ctx, th, grads, m, v, self.proj, self.tiles, self.out,
                             self.state, self.lr, lambda_ssim=self.lam)
            for t in range(self.T if allowed else 0):
                ci = self.next_camera(allowed)
                F = self.F[ci] if self.mode == "abcd" else None
                B = self.B[ci] if self.mode == "abcd" else None
                step(self.cams[ci], F, B, self.gt[ci], self.loss[t:t + 1], t + 1)
                if trace is not None:
                    trace(t, ci, th, grads, m, v, self.loss[t:t + 1])
        self.steps_done += self.T if allowed else 0
        self.update_frustum()                  # the block's Gaussians moved
        self.refresh(b)

    def stage_render(self, b, ci):
        """The composite the first step of block b's stage renders for camera ci (F over the
        block, with its halo, over B), fp32 RGBA; the parameters are left unchanged."""
        if self.mode == "abcd":
            self.composite(b)
        ths = self._stage_theta(b)
        cam = self.cams[ci]
        F = self.F[ci] if self.mode == "abcd" else None
        B = self.B[ci] if self.mode == "abcd" else None
        abcd_project(self.ctx, ths, cam, None, self.proj)
        abcd_bin_sort(self.ctx, self.proj, ths.n, cam, self.tiles)
        out = self.torch.empty(self.H, self.W, 4, device="cuda")
        abcd_render_composite_fwd(self.ctx, cam, None, self.proj, self.tiles, F, B, ABCD_F16,
                                  None, out, None)
        return out

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
                       cull_tau=0.01, overlap=1.0):
    """Section 3's comparison on a seeded synthetic scene (a 2x2x1 grid of side 5, SH degree
    0): full-scene training (one block, 4 T steps per cycle), ABCD and the ablated variant (4
    blocks, T steps each per cycle), the same number of steps in all three, against targets
    rendered from a perturbed copy of the scene; and ABCD with the camera-partition pairs
    culled at visible share cull_tau (Section 4), which trains each block on the cameras that
    see it, and ABCD with an overlapping boundary region of width `overlap` (Section 4).
    Returns {name: [eval loss after 0..cycles]}; the eval renders every layer."""
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
    for name, d, sd, mode, t, tau, ov in (
            ("full_scene", (1, 1, 1), 2 * side, "abcd", 4 * T, None, 0.0),
            ("abcd", dims, side, "abcd", T, None, 0.0),
            ("ablated", dims, side, "ablated", T, None, 0.0),
            ("abcd_culled", dims, side, "abcd", T, cull_tau, 0.0),
            ("abcd_overlap", dims, side, "abcd", T, None, overlap)):
        run = BCD(s.gaussians, d, origin, sd, s.cameras, targets, t, default_lr(2 * side),
                  mode=mode, seed=seed + 2, cull_tau=tau, overlap=ov)
        hist = [run.eval_loss()]
        for _ in range(cycles):
            run.cycle()
            hist.append(run.eval_loss())
        out[name] = hist
    return out
