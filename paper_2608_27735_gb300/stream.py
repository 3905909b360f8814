"""Out-of-core ABCD stages: the memory hierarchy of Section 2.

The parameters of every block and the cached renders of every camera-partition pair stay in
host memory (pinned) or, with a cache directory, on disk (the disk tier); the GPU holds only
the active block with its gradient and Adam moments, one workspace, a staging buffer of fixed
size for the frozen layers of one camera, two fp32 accumulators and two slots of one F/B pair
and one target.  None of these grows with the number of partitions or cameras, so the peak
device memory of a stage is O(1) in the scene's extent for a fixed partition size and image
resolution (Section 3).

A stage of block b:
  1. its parameters go to the device; the Adam moments start from zero;
  2. for every camera, F and B are folded from the frozen blocks' cached layers in the camera's
     depth order, the layers streamed through the staging buffer in pieces and folded into an
     fp32 accumulator (abcd_composite_fold_packed: the same result as folding them at once,
     bit for bit); the fp16 F and B go back to host memory;
  3. T steps, each on a sampled camera, with that camera's F, B and target copied into one of
     two device slots one step ahead (abcd_cache_fetch on the context's copy stream), so the
     copies overlap the step before (the "single image pair at a time" mode of Section 2);
  4. every camera's layer of block b is re-rendered into a packed layer and stored back;
  5. the parameters go back to host memory.
Host orchestration of the C ABI only: every operation on the data runs in libabcd's kernels.
"""
from __future__ import annotations

import os

import numpy as np

from . import (Context, FwdState, Gaussians, Projected, RefreshLayer, Tiles, TrainStep, TILE,
               abcd_assign_cells, abcd_cache_fetch, abcd_cache_release, abcd_cache_store,
               abcd_cache_sync, abcd_cache_wait, abcd_composite_fold_packed,
               abcd_partition_split, camera, visible_pairs, _torch)

BLOCK_TILE = (TILE, TILE, 4)          # one stored tile of a packed layer: 16 x 16 fp16 RGBA
MAX_PIECE_LAYERS = 64                 # layers folded per call (tile maps staged at once)


class LayerStore:
    """The cached packed layers of every (camera, block) pair: the tile map (int32 [tiles]) and
    the stored tiles (fp16 [count][16][16][4]).  In pinned host memory, or with `directory`, in
    one file per pair on disk (the disk tier), read back into pinned staging on use."""

    def __init__(self, n_tiles, directory=None):
        self.torch = _torch()
        self.n_tiles = int(n_tiles)
        self.dir = directory
        self.mem = {}
        if directory:
            os.makedirs(directory, exist_ok=True)

    def _path(self, ci, b):
        return os.path.join(self.dir, f"layer_c{ci}_b{b}.bin")

    def put(self, ci, b, tile_map, tiles):
        """tile_map: int32 host tensor [tiles]; tiles: fp16 host tensor [count][16][16][4]."""
        if self.dir:
            with open(self._path(ci, b), "wb") as f:
                f.write(np.int64(tiles.shape[0]).tobytes())
                f.write(tile_map.numpy().tobytes())
                f.write(tiles.numpy().tobytes())
        else:
            self.mem[ci, b] = (tile_map.pin_memory(), tiles.pin_memory())

    def get(self, ci, b):
        """(tile map, stored tiles) as pinned host tensors."""
        if not self.dir:
            return self.mem[ci, b]
        torch = self.torch
        with open(self._path(ci, b), "rb") as f:
            count = int(np.frombuffer(f.read(8), np.int64)[0])
            m = np.frombuffer(f.read(4 * self.n_tiles), np.int32)
            t = np.frombuffer(f.read(2 * count * TILE * TILE * 4), np.float16).reshape(count, *BLOCK_TILE)
        return (torch.from_numpy(m.copy()).pin_memory(), torch.from_numpy(t.copy()).pin_memory())

    def count(self, ci, b):
        if not self.dir:
            return int(self.mem[ci, b][1].shape[0])
        with open(self._path(ci, b), "rb") as f:
            return int(np.frombuffer(f.read(8), np.int64)[0])


class StreamingABCD:
    """Cyclic ABCD over the cells of a regular grid with the layers, F/B pairs and targets
    streamed through fixed device buffers.

    gaussians: scenegen.Gaussians of the whole scene; dims, origin, side: the grid; cameras:
    objects with R, t, fx, fy, cx, cy, width, height, position; targets: float32 [C][H][W][3];
    max_pairs: tile-pair capacity of the active block's lists; stage_tiles: capacity of the
    staging buffer in stored tiles (at least one full layer's tiles); cache_dir: put the cached
    layers on disk instead of in host memory."""

    def __init__(self, gaussians, dims, origin, side, cameras, targets, T, lr, max_pairs,
                 stage_tiles=None, device=0, seed=0, lambda_ssim=0.2, cache_dir=None):
        torch = _torch()
        self.torch, self.T, self.lam = torch, int(T), float(lambda_ssim)
        self.ctx = Context(device)
        self.dims = tuple(int(d) for d in dims)
        self.origin = [float(v) for v in origin]
        self.side = float(side)
        n_blocks = int(np.prod(self.dims))
        cells = abcd_assign_cells(gaussians.means, self.origin, self.side, self.dims)
        self.members = [np.nonzero(cells == b)[0] for b in range(n_blocks)]
        self.blocks = [b for b in range(n_blocks) if len(self.members[b])]
        # every block's parameters in pinned host memory
        self.host_theta = {b: [torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
                               for a in gaussians.subset(self.members[b]).arrays()]
                           for b in self.blocks}
        self.sh_degree = int(gaussians.sh_degree)
        self.n_max = max(len(self.members[b]) for b in self.blocks)
        self.cams_np = list(cameras)
        self.cams = [camera(c) for c in cameras]
        W, H = int(cameras[0].width), int(cameras[0].height)
        self.W, self.H = W, H
        tx, ty = (W + TILE - 1) // TILE, (H + TILE - 1) // TILE
        self.n_t = tx * ty
        self.stage_tiles = int(stage_tiles or 2 * self.n_t)
        assert self.stage_tiles >= self.n_t, "the staging buffer must hold one full layer"
        self.store = LayerStore(self.n_t, cache_dir)
        self.host_gt = torch.from_numpy(np.ascontiguousarray(targets, dtype=np.float32)).pin_memory()
        C = len(cameras)
        self.host_F = torch.empty(C, H, W, 4, dtype=torch.float16).pin_memory()
        self.host_B = torch.empty_like(self.host_F).pin_memory()
        self.order = {}
        for ci, c in enumerate(cameras):
            for b in range(n_blocks):
                f, bk = abcd_partition_split(self.dims, self.origin, self.side, c.position, b)
                self.order[ci, b] = (list(f), list(bk))
        self.lr = list(lr)
        self.rng = np.random.default_rng(seed)
        self.queue = []
        # ---- the device: fixed buffers, whatever the number of blocks and cameras
        dev = "cuda"
        f = lambda *s, dt=torch.float32: torch.zeros(*s, dtype=dt, device=dev)
        D = (self.sh_degree + 1) ** 2
        mk = lambda: Gaussians(f(self.n_max, 3), f(self.n_max, 3), f(self.n_max, 4), f(self.n_max),
                               f(self.n_max, D, 3), self.sh_degree)
        self.theta, self.grads, self.m, self.v = mk(), mk(), mk(), mk()
        self.ctx.reserve(self.n_max, max_pairs, W * H)
        self.proj = Projected.alloc(self.n_max)
        self.tiles = Tiles.alloc(max_pairs, W, H)
        self.out = f(H, W, 4)
        self.state = FwdState.alloc(W, H)
        self.loss = f(max(1, self.T))
        self.acc = f(H, W, 4)
        self.stage_buf = [f(self.stage_tiles, *BLOCK_TILE, dt=torch.float16) for _ in range(2)]
        self.stage_maps = [f(MAX_PIECE_LAYERS, self.n_t, dt=torch.int32) for _ in range(2)]
        self.slots = [dict(F=f(H, W, 4, dt=torch.float16), B=f(H, W, 4, dt=torch.float16),
                           gt=f(H, W, 3)) for _ in range(2)]
        self.ref_tiles = [f(self.n_t, *BLOCK_TILE, dt=torch.float16) for _ in range(2)]
        self.ref_maps = [f(self.n_t, dt=torch.int32) for _ in range(2)]
        self.ref_cnt = f(2, dt=torch.int32)
        # host staging of a refreshed layer on its way back
        self.back_tiles = torch.empty(self.n_t, *BLOCK_TILE, dtype=torch.float16).pin_memory()
        self.back_map = torch.empty(self.n_t, dtype=torch.int32).pin_memory()
        self.back_cnt = torch.empty(2, dtype=torch.int32).pin_memory()
        self.loss_host = torch.empty(max(1, self.T), dtype=torch.float32).pin_memory()
        # a0: pairs whose partition meets the camera's frustum (the others are transparent:
        # stored empty, not rendered, not trained on)
        self.frustum = np.zeros((C, n_blocks), bool)
        for b in self.blocks:                   # the initial cache: every block's layers
            self._load(b)
            self.refresh(b)

    # ---- pieces of a stage
    def _view(self, b):
        n = len(self.members[b])
        return (Gaussians(*(t[:n] for t in self.theta.tensors()), self.sh_degree),
                Gaussians(*(t[:n] for t in self.grads.tensors()), self.sh_degree),
                Gaussians(*(t[:n] for t in self.m.tensors()), self.sh_degree),
                Gaussians(*(t[:n] for t in self.v.tensors()), self.sh_degree))

    def _load(self, b):
        th, _, m, v = self._view(b)
        for dst, src in zip(th.tensors(), self.host_theta[b]):
            dst.copy_(src, non_blocking=True)
        for x in (m, v):
            for t in x.tensors():
                t.zero_()

    def _save(self, b):
        th = self._view(b)[0]
        for src, dst in zip(th.tensors(), self.host_theta[b]):
            dst.copy_(src, non_blocking=True)

    def refresh(self, b):
        """Block b's layer for every camera that sees it, rendered into a packed layer and
        stored (an empty layer for the others)."""
        th = self._view(b)[0]
        self.frustum[:, b] = visible_pairs(self.ctx, {b: th}, self.cams, self.dims, self.origin,
                                           self.side)[:, b]
        rl = RefreshLayer(self.ctx, th, self.proj, self.tiles)
        for ci, cam in enumerate(self.cams):
            if not self.frustum[ci, b]:
                self.store.put(ci, b, self.torch.full((self.n_t,), -1, dtype=self.torch.int32),
                               self.torch.empty(0, *BLOCK_TILE, dtype=self.torch.float16))
                continue
            rl(cam, self.ref_maps[0], self.ref_tiles[0], self.ref_cnt[0:1])
            self.back_cnt.copy_(self.ref_cnt, non_blocking=True)
            self.ctx.sync()
            n = int(self.back_cnt[0])
            self.back_map.copy_(self.ref_maps[0])
            self.back_tiles[:n].copy_(self.ref_tiles[0][:n])
            self.store.put(ci, b, self.back_map.clone(), self.back_tiles[:n].clone())

    def fold_fb(self, b):
        """F and B of every camera around block b, folded from the stored layers through the
        staging buffer, into host memory."""
        ctx = self.ctx
        k = 0                                      # staging buffer / copy slot in use
        for ci in range(len(self.cams)):
            keep = []                              # host buffers of queued copies stay alive
            front, back = self.order[ci, b]
            for side, dst in ((front, self.host_F[ci]), (back, self.host_B[ci])):
                out16 = self.slots[0]["F"]
                if not side:
                    out16.zero_()
                else:
                    # consecutive layers into pieces that fit the staging buffer
                    pieces, cur, used = [], [], 0
                    for q in side:
                        c = self.store.count(ci, q)
                        if cur and (used + c > self.stage_tiles or len(cur) == self.stage_maps[0].shape[0]):
                            pieces.append(cur)
                            cur, used = [], 0
                        cur.append(q)
                        used += c
                    pieces.append(cur)
                    for j, piece in enumerate(pieces):
                        buf, maps = self.stage_buf[k], self.stage_maps[k]
                        off, views_m, views_t = 0, [], []
                        for i, q in enumerate(piece):
                            hm, ht = self.store.get(ci, q)
                            keep.append((hm, ht))
                            abcd_cache_fetch(ctx, k, hm, maps[i])
                            c = int(ht.shape[0])
                            if c:
                                abcd_cache_fetch(ctx, k, ht, buf[off:off + c])
                            views_m.append(maps[i])
                            views_t.append(buf[off:] if c else buf)
                            off += c
                        abcd_cache_wait(ctx, k)
                        last = j == len(pieces) - 1
                        abcd_composite_fold_packed(ctx, views_m, views_t, self.W, self.H,
                                                   acc_in=self.acc if j else None,
                                                   acc_out=None if last else self.acc,
                                                   out16=out16 if last else None)
                        abcd_cache_release(ctx, k)
                        k = 1 - k
                abcd_cache_store(ctx, 0, out16, dst)
                abcd_cache_wait(ctx, 0)            # out16 is rewritten by the next fold
            if self.store.dir:
                abcd_cache_sync(ctx)               # the disk tier's staging copies are done
                keep.clear()
        abcd_cache_sync(ctx)

    def next_camera(self, allowed=None):
        """Shuffle without replacement over the allowed cameras, reshuffled when used up."""
        allowed = list(range(len(self.cams))) if allowed is None else list(allowed)
        self.queue = [ci for ci in self.queue if ci in allowed]
        if not self.queue:
            self.queue = [allowed[i] for i in self.rng.permutation(len(allowed))]
        return int(self.queue.pop())

    def stage(self, b, trace=None):
        """One stage of block b (see the module docstring).  trace, if given, is called after
        every step as trace(t, camera, theta, grads, m, v, loss) with the device tensors."""
        ctx = self.ctx
        self._load(b)
        self.fold_fb(b)
        th, gr, m, v = self._view(b)
        step = TrainStep(ctx, th, gr, m, v, self.proj, self.tiles, self.out, self.state, self.lr,
                         lambda_ssim=self.lam)
        allowed = [ci for ci in range(len(self.cams)) if self.frustum[ci, b]]
        order = [self.next_camera(allowed) for _ in range(self.T)] if allowed else []

        def fetch(k, ci):
            s = self.slots[k]
            abcd_cache_fetch(ctx, 2 + k, self.host_F[ci], s["F"])
            abcd_cache_fetch(ctx, 2 + k, self.host_B[ci], s["B"])
            abcd_cache_fetch(ctx, 2 + k, self.host_gt[ci], s["gt"])

        if order:
            fetch(0, order[0])
        for t, ci in enumerate(order):
            k = t % 2
            abcd_cache_wait(ctx, 2 + k)
            if t + 1 < len(order):
                fetch(1 - k, order[t + 1])         # starts once the step before has released it
            s = self.slots[k]
            step(self.cams[ci], s["F"], s["B"], s["gt"], self.loss[t:t + 1], t + 1)
            abcd_cache_release(ctx, 2 + k)
            if trace is not None:
                trace(t, ci, th, gr, m, v, self.loss[t:t + 1])
        self.loss_host.copy_(self.loss)
        self.refresh(b)
        self._save(b)
        ctx.sync()
        return self.loss_host[:len(order)].clone()

    def cycle(self):
        for b in self.blocks:
            self.stage(b)

    # ---- checkpoint / resume: every block's parameters and the cached layers on disk
    def save(self, directory):
        """Writes every block's parameters (one .npz per block) and, for an in-memory cache,
        every cached layer (the disk tier's files) under `directory`.  The Adam moments are
        not saved: every stage starts them from zero."""
        os.makedirs(directory, exist_ok=True)
        for b in self.blocks:
            np.savez(os.path.join(directory, f"theta_b{b}.npz"),
                     *[t.numpy() for t in self.host_theta[b]])
        disk = LayerStore(self.n_t, os.path.join(directory, "layers"))
        if self.store.dir != disk.dir:
            for ci in range(len(self.cams)):
                for b in self.blocks:
                    m, t = self.store.get(ci, b)
                    disk.put(ci, b, m, t)

    def load(self, directory):
        """Reads what save() wrote into this object (the same scene layout)."""
        for b in self.blocks:
            with np.load(os.path.join(directory, f"theta_b{b}.npz")) as z:
                for k, t in enumerate(self.host_theta[b]):
                    t.copy_(self.torch.from_numpy(z[f"arr_{k}"]))
        disk = LayerStore(self.n_t, os.path.join(directory, "layers"))
        for ci in range(len(self.cams)):
            for b in self.blocks:
                m, t = disk.get(ci, b)
                self.store.put(ci, b, m, t)

    def device_bytes(self):
        """Bytes of the device buffers this object holds (workspace included)."""
        torch = self.torch
        ts = list(self.theta.tensors()) + list(self.grads.tensors()) + list(self.m.tensors()) + \
            list(self.v.tensors()) + [self.proj.uv, self.proj.conic_opacity, self.proj.rgb,
                                      self.proj.depth, self.proj.radius, self.proj.tiles_touched,
                                      self.tiles.ids, self.tiles.ranges, self.tiles.count,
                                      self.out, self.state.A_T, self.state.n_last, self.loss,
                                      self.acc, self.ref_cnt, self.ctx.workspace] + \
            self.stage_buf + self.stage_maps + self.ref_tiles + self.ref_maps + \
            [x for s in self.slots for x in s.values()]
        return int(sum(t.numel() * t.element_size() for t in ts if isinstance(t, torch.Tensor)))
