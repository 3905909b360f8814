#!/usr/bin/env python
"""Benchmark of the ABCD hot path on the scene-scale workload.

Workload (one bench step = one ABCD stage, Section 2): a 4x4x2 grid of partitions (side 5)
with 100,000 Gaussians each (SH degree 3, 3.2M in total), 200 cameras at 1237x822 on a ring
with height jitter; the active block is cell (1, 1, 0).  A stage
  1. composites, for every camera observing the active partition, the cached fp16 renders of
     the frozen partitions into F and B in that camera's depth order (K1);
  2. runs T = 500 active-block steps, each on a sampled camera: project (K2), bin + sort
     (K3/K4), render + composite F over A over B (K5), L1 + 0.2 D-SSIM loss (K6), backward into
     the active block (K7, K8) and Adam (K9);
  3. refreshes the active partition's cached renders for every observing camera (K10).
value = active-block steps per second (T x stages / time), inputs resident in HBM.
e2e = the same metric through the C ABI with the stage's inputs in pinned host memory: the
cached layers, targets and active parameters are copied in and the refreshed layers,
parameters and losses copied out inside the timed region, every stage.
Inputs are synthetic (paper_2608_27735_gb300.scenegen), shaped like the paper's scenes.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "ABCD active-block steps/s @1237x822, 100k Gaussians; % of roofline"
UNIT = "steps/s"
ACTIVE_CELL = (1, 1, 0)
LR = [1.6e-4 * 15.0, 5e-3, 1e-3, 0.025, 2.5e-3, 2.5e-3 / 20]   # means lr scaled by the scene extent
REFRESH_STREAMS = 8         # concurrent cache-refresh pipelines (contexts with their own streams)
FWD_FLOP_PER_PAIR = 25      # per (pixel, list entry) walked: offset, sigma, alpha, tests, blend
BWD_FLOP_PER_PAIR = 68      # recompute + d alpha + colour, opacity, mean and conic terms
LOSS_FLOP_PER_PX = 1000     # five 11-tap windows twice (separable), SSIM terms, 3 channels


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3, help="timed ABCD stages")
    ap.add_argument("--warmup", type=int, default=3, help="untimed ABCD stages")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--T", type=int, default=500, help="active-block steps per stage")
    ap.add_argument("--cams", type=int, default=200)
    ap.add_argument("--per-cell", type=int, default=100_000)
    ap.add_argument("--width", type=int, default=1237)
    ap.add_argument("--height", type=int, default=822)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the measurements of the other workload configurations")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sample-every", type=int, default=10, help="per-op event sampling stride")
    return ap.parse_args(argv)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(ms, world):
    """The slowest rank's time: replicas report the whole job's throughput over it."""
    if world <= 1:
        return float(ms)
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(ms)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_value(stages, T, world, ms):
    """Active-block steps/s of the whole job: every rank runs `stages` stages of T steps."""
    return stages * T * world / (ms / 1e3)


# ---------------------------------------------------------------------------------------
# clocks during the timed region

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.proc = None
        self.device = device

    def start(self):
        import torch
        sel = []
        try:
            p = torch.cuda.get_device_properties(self.device)
            bus = f"{p.pci_domain_id:08x}:{p.pci_bus_id:02x}:{p.pci_device_id:02x}.0"
            sel = ["-i", bus]
        except Exception:
            pass
        try:
            self.proc = subprocess.Popen(["nvidia-smi", *sel, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for nm, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": float(max(mx)) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------------------
# the workload on the GPU

class Stage:
    """Device-resident scene-scale ABCD stage driven through the C ABI."""

    def __init__(self, args, device, seed=1003, log=print):
        import torch
        import paper_2608_27735_gb300 as ab
        from paper_2608_27735_gb300 import scenegen as sg
        self.torch, self.ab, self.sg = torch, ab, sg
        self.args = args
        self.dev = device
        t0 = time.time()
        scene = sg.scene_scale(seed=seed, per_cell=args.per_cell, width=args.width,
                               height=args.height, n_cams=args.cams)
        self.scene = scene
        g = scene.gaussians
        grid = scene.grid
        self.W, self.H = args.width, args.height
        self.cells = ab.abcd_assign_cells(g.means, grid.origin, grid.side, grid.dims)
        gx, gy, _ = grid.dims
        self.active = ACTIVE_CELL[0] + gx * (ACTIVE_CELL[1] + gy * ACTIVE_CELL[2])
        self.n_parts = grid.n_cells
        self.ctx = ab.Context(device)
        self.stream = self.ctx.stream
        log(f"[bench] scene generated in {time.time() - t0:.1f}s ({g.n} Gaussians)")
        # per-partition parameters on the device (for the initial cache only)
        self.part_idx = [np.nonzero(self.cells == p)[0] for p in range(self.n_parts)]
        n_max = max(len(ix) for ix in self.part_idx)
        self.cams = [ab.camera(c) for c in scene.cameras]
        self.splits = []
        for c in scene.cameras:
            f, b = ab.abcd_partition_split(grid.dims, grid.origin, grid.side, c.position, self.active)
            self.splits.append((list(f), list(b)))
        npx = self.W * self.H
        self.ctx.reserve(max(n_max, 1), 16_000_000, npx)
        self.theta = ab.Gaussians.from_numpy(g.subset(self.part_idx[self.active]), device)
        self.n = self.theta.n
        self.grads = ab.Gaussians.zeros_like(self.theta)
        self.m = ab.Gaussians.zeros_like(self.theta)
        self.v = ab.Gaussians.zeros_like(self.theta)
        self.proj = ab.Projected.alloc(n_max, device)
        self.out = torch.empty(self.H, self.W, 4, device=device)
        self.state = ab.FwdState.alloc(self.W, self.H, device)
        self.loss = torch.zeros(args.T, device=device)
        C = len(self.cams)
        # tile-list capacity: pair counts K of every (partition, camera) render, +25%
        self.tiles = ab.Tiles.alloc(64_000_000, self.W, self.H, device)
        self.ctx.reserve(max(n_max, 1), 64_000_000, npx)
        self.part_dev = {}
        tgt = sg.perturbed(g, grid.side, seed=seed + 1)
        self.tgt_dev = [ab.Gaussians.from_numpy(tgt.subset(self.part_idx[p]), device)
                        for p in range(self.n_parts)]
        ks, ks_active = [], []
        for p in range(self.n_parts):
            th = ab.Gaussians.from_numpy(g.subset(self.part_idx[p]), device)
            for src in (th, self.tgt_dev[p]):
                for ci in range(C):
                    ab.abcd_project(self.ctx, src, self.cams[ci], None, self.proj)
                    ab.abcd_bin_sort(self.ctx, self.proj, src.n, self.cams[ci], self.tiles)
                    ks.append(self.tiles.count.clone())
                    if p == self.active and src is th:
                        ks_active.append(ks[-1])
        try:
            self.ctx.sync()
        except ab.AbcdError:
            self.ctx.clear_status()
            self.ctx.sync()
        kmax = int(torch.stack(ks).max().item())
        self.k_mean = float(torch.stack(ks_active).double().mean().item())
        cap = int(kmax * 1.25) + 1024
        self.ctx.reserve(max(n_max, 1), cap, npx)
        self.tiles = ab.Tiles.alloc(cap, self.W, self.H, device)
        log(f"[bench] active block n={self.n}, pairs K mean {self.k_mean:.0f}; max over all "
            f"partitions {kmax}, capacity {cap}")
        # cache of fp16 premultiplied renders, one per (camera, partition), in the packed
        # (tile-sparse) format: per camera, the frozen partitions' stored tiles back to back
        # (layer p at block offset self.pk_off[ci][p]) and the active partition's layer at
        # full capacity (the refresh rewrites it); tile maps for all layers
        t1 = time.time()
        P, a = self.n_parts, self.active
        self.n_t = ((self.W + 15) // 16) * ((self.H + 15) // 16)
        self.pk_map = torch.empty(C, P, self.n_t, dtype=torch.int32, device=device)
        self.pk_active = torch.empty(C, self.n_t, 16, 16, 4, dtype=torch.float16, device=device)
        self.pk_count = torch.zeros(C, P, dtype=torch.int32, device=device)
        ths = [ab.Gaussians.from_numpy(g.subset(self.part_idx[p]), device) for p in range(P)]
        # a0: the visible camera-partition pairs (frustum filter on each partition's cell and
        # 3-sigma box); the cameras that observe the active partition train it
        self.vis_pairs = ab.visible_pairs(self.ctx, {p: ths[p] for p in range(P)}, scene.cameras,
                                          grid.dims, grid.origin, grid.side)
        self.observing = [ci for ci in range(C) if self.vis_pairs[ci, a]]
        self.runs_mean = self.count_runs(self.theta, 4)
        log(f"[bench] visible camera-partition pairs {int(self.vis_pairs.sum())} of {C * P}; "
            f"{len(self.observing)} cameras observe the active partition")
        tmp = torch.empty(P, self.n_t, 16, 16, 4, dtype=torch.float16, device=device)
        self.pk_frozen, self.pk_off = [], []
        for ci in range(C):
            for p in range(P):
                self.render_packed(ths[p], ci, tmp[p] if p != a else self.pk_active[ci], p)
            cnt = self.pk_count[ci].cpu().numpy()
            off, run = [0] * P, 0
            for p in range(P):
                if p != a:
                    off[p], run = run, run + int(cnt[p])
            buf = torch.empty(max(run, 1), 16, 16, 4, dtype=torch.float16, device=device)
            for p in range(P):
                if p != a and cnt[p]:
                    buf[off[p]:off[p] + int(cnt[p])].copy_(tmp[p][:int(cnt[p])])
            self.pk_frozen.append(buf)
            self.pk_off.append(off)
        del tmp, ths
        self.ctx.sync()
        stored = sum(int(b.numel()) * 2 for b in self.pk_frozen)
        self.cache_bytes = stored
        log(f"[bench] cache of {C}x{P} layers: {stored / 1e9:.1f} GB of stored tiles for the frozen "
            f"partitions ({100.0 * stored / (C * (P - 1) * self.n_t * 2048):.0f}% of the tiles) "
            f"in {time.time() - t1:.1f}s")
        # targets: renders of the seed-perturbed scene
        t1 = time.time()
        self.gt = torch.empty(C, self.H, self.W, 3, device=device)
        self.render_targets()
        log(f"[bench] targets in {time.time() - t1:.1f}s")
        self.F = torch.empty(C, self.H, self.W, 4, dtype=torch.float16, device=device)
        self.B = torch.empty_like(self.F)
        # the cache refresh renders every observing camera independently: REFRESH_STREAMS side
        # contexts (own stream, workspace and buffers) take the cameras in turn, forked from and
        # joined back to the main stream with events
        self.side = []
        for _ in range(REFRESH_STREAMS):
            sctx = ab.Context(device, stream=torch.cuda.Stream(device))
            sctx.reserve(max(n_max, 1), cap, npx)
            self.side.append(dict(ctx=sctx, proj=ab.Projected.alloc(n_max, device),
                                  tiles=ab.Tiles.alloc(cap, self.W, self.H, device)))
        self.rng = np.random.default_rng(seed + 7)
        self.order = []
        self.step_count = 0
        self.events = {}
        self.pairs_sample = []
        self.sample_every = max(1, args.sample_every)

    def render_layer(self, th, ci, dst, w=None):
        ab = self.ab
        ctx, proj, tiles = (self.ctx, self.proj, self.tiles) if w is None else (w["ctx"], w["proj"], w["tiles"])
        ab.abcd_project(ctx, th, self.cams[ci], None, proj)
        ab.abcd_bin_sort(ctx, proj, th.n, self.cams[ci], tiles)
        ab.abcd_render_composite_fwd(ctx, self.cams[ci], None, proj, tiles, refresh_f16=dst)

    def render_packed(self, th, ci, dst, p, w=None, map_dst=None, cnt_dst=None):
        """K2-K4 and K10 into the packed layer dst (tile map and count of partition p, or into
        map_dst / cnt_dst), in one library call."""
        ab = self.ab
        holder = self.__dict__ if w is None else w
        fn = holder.get("_refresh") if th is self.theta else None
        if fn is None:
            ctx, proj, tiles = (self.ctx, self.proj, self.tiles) if w is None else (w["ctx"], w["proj"], w["tiles"])
            fn = ab.RefreshLayer(ctx, th, proj, tiles)
            if th is self.theta:
                holder["_refresh"] = fn
        fn(self.cams[ci], self.pk_map[ci, p] if map_dst is None else map_dst, dst,
           self.pk_count[ci, p:p + 1] if cnt_dst is None else cnt_dst)

    def packed_layers(self, ci):
        """Tile maps and packed data of camera ci's layers (None at the active partition)."""
        P, a = self.n_parts, self.active
        maps = [self.pk_map[ci, p] for p in range(P)]
        data = [self.pk_frozen[ci][self.pk_off[ci][p]:] if p != a else None for p in range(P)]
        maps[a] = None
        return maps, data

    def render_targets(self):
        torch, ab = self.torch, self.ab
        # full-scene render of the perturbed scene, partition by partition, composited in
        # each camera's depth order (associativity of 'over')
        tmp = torch.empty(self.n_parts, self.H, self.W, 4, dtype=torch.float16, device=self.dev)
        full = torch.empty(self.H, self.W, 4, dtype=torch.float32, device=self.dev)
        th = self.tgt_dev
        for ci in range(len(self.cams)):
            for p in range(self.n_parts):
                self.render_layer(th[p], ci, tmp[p])
            f, b = self.splits[ci]
            order = f + [self.active] + b
            ab.abcd_composite_cache(self.ctx, [tmp[p] for p in range(self.n_parts)], order,
                                    self.n_parts, self.W, self.H, full, None, ab.ABCD_F16,
                                    ab.ABCD_F32)
            self.gt[ci].copy_(full[..., :3])
        self.ctx.sync()
        self.tgt_dev = None

    def count_runs(self, th, n_cams):
        """Mean number of (Gaussian, tile row) runs of the active block over a few observing
        cameras: the distinct ids of each tile row's lists (one run per Gaussian and row)."""
        ab = self.ab
        tx, ty = (self.W + 15) // 16, (self.H + 15) // 16
        out = []
        for ci in list(self.observing)[:n_cams]:
            ab.abcd_project(self.ctx, th, self.cams[ci], None, self.proj)
            ab.abcd_bin_sort(self.ctx, self.proj, th.n, self.cams[ci], self.tiles)
            self.ctx.sync()
            K = int(self.tiles.count.item())
            rg = self.tiles.ranges[:tx * ty].cpu().numpy().astype(np.int64)
            ids = self.tiles.ids[:K].cpu().numpy()
            out.append(sum(len(np.unique(ids[rg[y * tx, 0]:rg[y * tx + tx - 1, 1]]))
                           for y in range(ty)))
        return float(np.mean(out)) if out else 0.0

    # ---- timing helpers
    def _mark(self, name, sampled, fn, *a, **k):
        if sampled:
            s = torch_event(self.torch, self.stream)
            fn(*a, **k)
            e = torch_event(self.torch, self.stream)
            self.events.setdefault(name, []).append((s, e))
        else:
            fn(*a, **k)

    def next_camera(self):
        if not self.order:
            self.order = list(self.rng.permutation(self.observing))
        return int(self.order.pop())

    # ---- the three parts of a stage
    def composite_all(self):
        """K1 for every observing camera.  The cameras' folds are independent, so they run on
        the side contexts' streams in turn (forked from and joined back to the stage stream with
        events, as the refresh does); the phase is timed as a whole."""
        torch = self.torch
        s = torch_event(torch, self.stream)
        for w in self.side:
            w["ctx"].stream.wait_event(s)
        for j, ci in enumerate(self.observing):
            self.composite_one(ci, ctx=self.side[j % len(self.side)]["ctx"])
        for w in self.side:
            self.stream.wait_event(torch_event(torch, w["ctx"].stream))
        e = torch_event(torch, self.stream)
        self.events.setdefault("composite_phase", []).append((s, e))

    def composite_one(self, ci, sampled=False, ctx=None):
        if not hasattr(self, "_pk_tables"):
            self._pk_tables = {}
        pl = self._pk_tables.get(ci)
        if pl is None:
            f, b = self.splits[ci]
            maps, data = self.packed_layers(ci)
            pl = self._pk_tables[ci] = self.ab.PackedLayers(maps, data, f + [self.active] + b, len(f))
        self._mark("composite", sampled, self.ab.abcd_composite_cache_packed_tables,
                   self.ctx if ctx is None else ctx, pl, self.W, self.H, self.F[ci], self.B[ci])

    def step(self, t, stage_step):
        ab = self.ab
        ci = self.next_camera()
        cam = self.cams[ci]
        smp = (self.step_count % self.sample_every) == 0
        self.step_count += 1
        if not smp:
            # the whole step in one call (the sampled steps below time each kernel)
            if not hasattr(self, "_train"):
                self._train = ab.TrainStep(self.ctx, self.theta, self.grads, self.m, self.v,
                                           self.proj, self.tiles, self.out, self.state, LR)
            self._train(cam, self.F[ci], self.B[ci], self.gt[ci], self.loss[t:t + 1], stage_step + 1)
            return
        self._mark("project", smp, ab.abcd_project, self.ctx, self.theta, cam, None, self.proj)
        self._mark("bin_sort", smp, ab.abcd_bin_sort, self.ctx, self.proj, self.n, cam, self.tiles)
        self._mark("render_fwd", smp, ab.abcd_render_composite_fwd, self.ctx, cam, None, self.proj,
                   self.tiles, self.F[ci], self.B[ci], ab.ABCD_F16, None, self.out, self.state)
        self._mark("loss", smp, ab.abcd_loss, self.ctx, self.out, self.gt[ci], self.W, self.H, 0.2,
                   self.loss[t:t + 1], self.ctx_dl())
        self._mark("render_bwd", smp, ab.abcd_render_backward, self.ctx, cam, None, self.proj,
                   self.tiles, self.F[ci], self.B[ci], ab.ABCD_F16, None, self.state, self.ctx_dl(),
                   self.n, self.ctx_g2d())
        self._mark("project_bwd", smp, ab.abcd_project_backward, self.ctx, self.theta, cam, None,
                   self.ctx_g2d(), self.grads)
        self._mark("adam", smp, ab.abcd_adam_active, self.ctx, self.theta, self.grads, self.m,
                   self.v, LR, 0.9, 0.999, 1e-15, stage_step + 1)
        if smp:
            self.pairs_sample.append(self.state.n_last.sum(dtype=self.torch.int64))

    def ctx_dl(self):
        if not hasattr(self, "_dl"):
            self._dl = self.torch.empty(self.H, self.W, 3, device=self.dev)
        return self._dl

    def ctx_g2d(self):
        if not hasattr(self, "_g2d"):
            self._g2d = self.torch.empty(self.n, 9, device=self.dev)
        return self._g2d

    def refresh_all(self):
        torch = self.torch
        s = torch_event(torch, self.stream)
        for w in self.side:
            w["ctx"].stream.wait_event(s)
        for j, ci in enumerate(self.observing):
            self.render_packed(self.theta, ci, self.pk_active[ci], self.active,
                               self.side[j % len(self.side)])
        for w in self.side:
            self.stream.wait_event(torch_event(torch, w["ctx"].stream))
        e = torch_event(torch, self.stream)
        # per camera: the phase's time over its cameras (they run REFRESH_STREAMS at a time)
        self.events.setdefault("refresh_phase", []).append((s, e))

    def launches(self):
        return self.ctx.launches() + sum(w["ctx"].launches() for w in self.side)

    def run_stage(self):
        for x in (self.m, self.v):          # Adam state starts from zero every stage
            for tns in x.tensors():
                tns.zero_()
        self.composite_all()
        for t in range(self.args.T):
            self.step(t, t)
        self.refresh_all()

    def reset_events(self):
        self.events = {}
        self.pairs_sample = []


def torch_event(torch, stream):
    e = torch.cuda.Event(enable_timing=True)
    e.record(stream)
    return e


def algorithmic(st: Stage, name, avg_ms, pairs_mean):
    """(bound, achieved, unit, peak_key) of one op from its algorithmic work per launch."""
    npx = st.W * st.H
    n = st.n
    D = 16
    if name == "render_fwd":
        return "alu", FWD_FLOP_PER_PAIR * pairs_mean / (avg_ms * 1e-3) / 1e12, "TFLOP/s"
    if name == "render_bwd":
        return "alu", BWD_FLOP_PER_PAIR * pairs_mean / (avg_ms * 1e-3) / 1e12, "TFLOP/s"
    if name == "loss":
        return "alu", LOSS_FLOP_PER_PX * npx / (avg_ms * 1e-3) / 1e12, "TFLOP/s"
    if name == "composite":
        # stored tiles of the frozen layers and their tile maps read, F and B written
        C = len(st.cams)
        byts = st.cache_bytes / C + (st.n_parts - 1) * st.n_t * 4 + 2 * 8 * npx
        return "hbm", byts / (avg_ms * 1e-3) / 1e9, "GB/s"
    P = 4 * PARAM_FLOATS(D)     # bytes of one Gaussian's parameters (236 at SH degree 3)
    if name == "adam":
        return "hbm", 7 * P * n / (avg_ms * 1e-3) / 1e9, "GB/s"
    if name == "project":
        return "hbm", (P + 52) * n / (avg_ms * 1e-3) / 1e9, "GB/s"
    if name == "project_bwd":
        return "hbm", (2 * P + 36) * n / (avg_ms * 1e-3) / 1e9, "GB/s"
    if name == "bin_sort":
        # keys and rectangles 20 B per Gaussian, four depth passes over 8-B items (16 B each);
        # runs: 8 B emitted, one row pass (16 B), 8 B read and a 4-B id written per pair by
        # the placement.  The working set stays in L2 and the passes are latency-bound, so the
        # HBM copy rate is a yardstick here, not the bound.
        K, R = st.k_mean, st.runs_mean
        byts = 20 * n + 4 * 16 * n + 8 * R + 16 * R + 8 * R + 4 * K
        return "latency", byts / (avg_ms * 1e-3) / 1e9, "GB/s"
    return None


def PARAM_FLOATS(D):
    """Floats per Gaussian: mean 3, log-scale 3, quaternion 4, opacity logit 1, SH 3 D."""
    return 3 + 3 + 4 + 1 + 3 * D


def measured_alu_peaks(device):
    """fp32 FMA and ex2.approx peaks measured on this device by the library's microbenchmark
    (SM count read from the device, CUDA events, no clock changes)."""
    import paper_2608_27735_gb300 as ab
    p = ab.abcd_measure_alu_peaks(device)
    p["fp32_tflops"] = max(p["ffma_tflops"], p["ffma2_tflops"])
    return p


def load_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return None


def profile_traffic(kernel):
    """DRAM bytes per launch from the committed ncu summary of `kernel`, or None if the
    summary is missing or the kernel's source changed since it was captured."""
    path = os.path.join(ROOT, "profiles", f"{kernel}.md")
    if not os.path.exists(path):
        return None
    txt = open(path).read()
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    h = re.search(r"source_sha256:\s*([0-9a-f]+)\s+(\S+)", txt)
    if not m or not h:
        return None
    src = os.path.join(ROOT, h.group(2))
    if not os.path.exists(src):
        return None
    if hashlib.sha256(open(src, "rb").read()).hexdigest() != h.group(1):
        return None
    return float(m.group(1))


def op_kernel_names():
    return {"render_fwd": "render_fwd_kernel", "render_bwd": "render_bwd_kernel",
            "loss": "ssim_fwd_kernel", "composite": "composite_kernel", "adam": "adam_kernel",
            "project": "project_fwd_kernel", "project_bwd": "project_bwd_kernel",
            "bin_sort": "binsort"}


# ---------------------------------------------------------------------------------------

def run_ours(args):
    import torch
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    log = (lambda *a: print(*a, file=sys.stderr, flush=True))
    import paper_2608_27735_gb300 as ab
    ab.build()
    st = Stage(args, local, log=log)
    for _ in range(args.warmup):
        st.run_stage()
    st.ctx.sync()
    st.reset_events()
    peaks = load_peaks()
    alu = measured_alu_peaks(local)
    log(f"[bench] measured fp32 FMA {alu['ffma_tflops']:.1f} TFLOP/s (FFMA2 {alu['ffma2_tflops']:.1f}), "
        f"ex2 {alu['ex2_tops']:.2f} T/s on {alu['sms']} SMs")

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    # ---- device-resident timed region
    clk = ClockSampler(local)
    barrier()
    torch.cuda.synchronize()
    clk.start()
    time.sleep(0.3)
    l0 = st.launches()
    torch.cuda.nvtx.range_push("abcd_timed")
    e0 = torch_event(torch, st.stream)
    h0 = time.perf_counter()
    for _ in range(args.steps):
        st.run_stage()
    host_ms = (time.perf_counter() - h0) * 1e3
    e1 = torch_event(torch, st.stream)
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    log(f"[bench] host issue time {host_ms / args.steps:.1f} ms per stage")
    barrier()
    launches = st.launches() - l0
    clocks = clk.stop()
    st.ctx.sync()
    ms = e0.elapsed_time(e1)
    ms = max_over_ranks(ms, world)
    value = replica_value(args.steps, args.T, world, ms)
    # per-op breakdown from the sampled events
    ops = {}
    for name, evs in st.events.items():
        ts = [s.elapsed_time(e) for s, e in evs]
        if name in ("refresh_phase", "composite_phase"):
            # per camera: the phase's time over its cameras (they run REFRESH_STREAMS at a time)
            ops[name.split("_")[0]] = dict(calls=len(ts), avg_ms=float(np.mean(ts)) / len(st.observing))
        else:
            ops[name] = dict(calls=len(ts), avg_ms=float(np.mean(ts)))
    per_stage = {"project": args.T, "bin_sort": args.T, "render_fwd": args.T, "loss": args.T,
                 "render_bwd": args.T, "project_bwd": args.T, "adam": args.T,
                 "composite": len(st.observing), "refresh": len(st.observing)}
    share = {k: ops[k]["avg_ms"] * per_stage[k] * args.steps / ms for k in ops}
    pairs_mean = float(torch.stack(st.pairs_sample).double().mean().item()) if st.pairs_sample else 0.0
    single = [k for k in ops if k not in ("bin_sort", "refresh")]
    dom = max(single, key=lambda k: share[k])
    hbm_peak = peaks["hbm_gbs"] if peaks else 6800.0
    hbm_note = "of measured (HBM copy, MEASURED_PEAKS.json)" if peaks else "of fallback"
    alu_note = (f"of measured (fp32 FMA microbenchmark on {alu['sms']} SMs: FFMA "
                f"{alu['ffma_tflops']:.1f}, FFMA2 {alu['ffma2_tflops']:.1f} TFLOP/s; the larger)")

    def roof(name):
        r = algorithmic(st, name, ops[name]["avg_ms"], pairs_mean)
        if r is None:
            return None
        bound, achieved, unit = r
        peak, note = ((hbm_peak, hbm_note) if bound == "hbm" else
                      (hbm_peak, "HBM copy rate as a yardstick: " + hbm_note) if bound == "latency"
                      else (alu["fp32_tflops"], alu_note))
        return dict(bound=bound, achieved=round(achieved, 3), peak=round(peak, 1), unit=unit,
                    frac=round(achieved / peak, 4), peak_source=note)

    rf = roof(dom)
    kname = op_kernel_names()[dom]
    roofline = dict(rf, traffic=profile_traffic(kname), kernel=kname,
                    algorithmic_per_launch=(f"{pairs_mean:.0f} pixel-list pairs" if dom.startswith("render")
                                            else None))
    per_kernel = {k: roof(k) for k in ops if k != "refresh"}
    # ---- end to end through the C ABI with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(st, args, world, barrier)
    streaming = None
    if not args.no_e2e:
        streaming = run_streaming(st, args, world, barrier)
    visibility = run_visibility(st)
    quality = None
    if rank == 0 and not args.no_e2e:
        # Section 3's comparison on a small seeded scene (about a second of GPU time)
        from paper_2608_27735_gb300.bcd import quality_experiment
        h = quality_experiment()
        quality = {k: [round(x, 5) for x in v] for k, v in h.items()}
        quality["note"] = ("eval loss (L1 + 0.2 D-SSIM of the full composited render, mean over 8 "
                           "cameras) after 0..3 cycles; 2x2x1 grid, 4000 Gaussians, equal step "
                           "counts; full_scene = one block; abcd_culled = camera-partition pairs "
                           "below a 1% visible share dropped; abcd_overlap = overlapping "
                           "boundary region of width 1 (a fifth of a cell)")
    configs = None
    if not args.no_configs:
        del st.pk_frozen, st.F, st.B, st.gt        # make room: the stage is measured
        torch.cuda.empty_cache()
        configs = {}
        for name, fn in (("cache_sweep_64_layers_1080p", run_cache_sweep),
                         ("stress_2M_1080p", run_stress),
                         ("grid_3x3x3_20k_640x480_stage", run_medium_stage)):
            t0 = time.time()
            configs[name] = fn(local)
            log(f"[bench] {name}: {configs[name]} ({time.time() - t0:.1f}s)")
        cs = configs["cache_sweep_64_layers_1080p"]
        cs["hbm_frac"] = round(cs["gbs"] / hbm_peak, 4)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args, log)
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded scenegen, shaped like the paper's 200-camera grid scenes)",
        "config": stage_config(args, st.n, world),
        "pairs_mean": round(st.k_mean),
        "runs_mean": round(st.runs_mean),
        "roofline": roofline,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "streaming_one_fb_pair": streaming,
        "bcd_quality": quality,
        "visibility_culling": visibility,
        "frustum": {"pairs": int(st.vis_pairs.size), "visible_pairs": int(st.vis_pairs.sum()),
                    "observing_cameras": len(st.observing),
                    "note": "a camera-partition pair is kept when the partition's cell united "
                            "with its Gaussians' 3-sigma box meets the guard-widened view "
                            "frustum (abcd_block_bounds, abcd_pair_visible); ring cameras "
                            "facing the grid see every partition"},
        "gpu_launches": int(launches),
        "clocks": clocks,
        "ops": {k: {"avg_ms": round(v["avg_ms"], 4), "share": round(share[k], 4)} for k, v in ops.items()},
        "rooflines": per_kernel,
        "configs": configs,
        "alu_peaks": {k: (round(v, 3) if isinstance(v, float) else v) for k, v in alu.items()},
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


TAU_VISIBLE = 1e-3


# ---------------------------------------------------------------------------------------
# the other workload configurations, measured after the headline stage (each bounded to
# seconds of GPU time)

def run_cache_sweep(device, n_cams=200, L=64, width=1920, height=1080, sets=16, seed=404):
    """K1 on the cache compositing sweep: per camera 64 fp16 premultiplied layers at 1080p in a
    random depth order, folded into F and B for the split at every position 1..63; 16 distinct
    layer sets (17 GB, far more than the L2) cycled over the 200 cameras with a fresh order
    each.  GB/s of algorithmic bytes ((L - 1) layers read, F and B written, per split)."""
    import torch
    import paper_2608_27735_gb300 as ab
    ctx = ab.Context(device)
    P = width * height
    g = torch.Generator(device=f"cuda:{device}")
    g.manual_seed(seed)
    layer_sets = []
    for _ in range(sets):
        a = torch.rand(L, height, width, 1, device=device, generator=g)
        rgb = torch.rand(L, height, width, 3, device=device, generator=g) * a
        layer_sets.append(torch.cat([rgb, a], -1).half())
        del a, rgb
    F = torch.empty(height, width, 4, dtype=torch.float16, device=device)
    B = torch.empty_like(F)
    rng = np.random.default_rng(seed)
    orders = [list(rng.permutation(L)) for _ in range(n_cams)]
    tables = []
    for ci in range(n_cams):
        st = layer_sets[ci % sets]
        tables.append([st[k] for k in range(L)])
    def sweep(cams):
        for ci in cams:
            for split in range(1, L):
                lay = list(tables[ci])
                lay[orders[ci][split]] = None
                ab.abcd_composite_cache(ctx, lay, orders[ci], split, width, height, F, B)
    sweep(range(2))
    torch.cuda.synchronize()
    e0 = torch_event(torch, ctx.stream)
    sweep(range(n_cams))
    e1 = torch_event(torch, ctx.stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    per = (L - 1) * 8 * P + 2 * 8 * P
    calls = n_cams * (L - 1)
    gbs = calls * per / (ms * 1e-3) / 1e9
    del layer_sets, tables
    torch.cuda.empty_cache()
    return {"workload": f"{L} fp16 RGBA layers {width}x{height} per camera, {n_cams} cameras, "
                        f"splits 1..{L - 1}, {sets} distinct layer sets ({sets * L * 8 * P / 1e9:.1f} GB)",
            "calls": calls, "ms": round(ms, 1), "us_per_split": round(1e3 * ms / calls, 2),
            "algorithmic_bytes_per_split": per, "gbs": round(gbs, 1), "kernel": "composite_kernel"}


def run_stress(device, n=2_000_000, width=1920, height=1080, n_cams=200, sampled=12, seed=505):
    """The stress block: 2M Gaussians (SH 3) from a 16-blob mixture, one dense block seen by 200
    ring cameras at 1920x1080; per sampled camera one forward + backward step (project, bin +
    sort, render, L1 + 0.2 D-SSIM against a target, backward to the parameters), timed with
    events; list statistics from the tile ranges."""
    import torch
    import paper_2608_27735_gb300 as ab
    from paper_2608_27735_gb300 import scenegen as sg
    g = sg.mixture_block(n, 20.0, 16, 3, seed=seed)
    cams_np = sg.ring_cameras(n_cams, 30.0, np.zeros(3), width, height, seed=seed, height_jitter=2.0)
    cams = [ab.camera(c) for c in cams_np]
    ctx = ab.Context(device)
    theta = ab.Gaussians.from_numpy(g)
    grads = ab.Gaussians.zeros_like(theta)
    proj = ab.Projected.alloc(n)
    cap = 450_000_000
    ctx.reserve(n, cap, width * height)
    tiles = ab.Tiles.alloc(cap, width, height)
    out = torch.empty(height, width, 4, device=device)
    state = ab.FwdState.alloc(width, height)
    gt = torch.rand(height, width, 3, device=device)
    loss = torch.zeros(sampled, device=device)
    pick = list(range(0, n_cams, max(1, n_cams // sampled)))[:sampled]
    def step(k, ci):
        ab.abcd_project(ctx, theta, cams[ci], None, proj)
        ab.abcd_bin_sort(ctx, proj, n, cams[ci], tiles)
        ab.abcd_render_composite_fwd(ctx, cams[ci], None, proj, tiles, None, None, ab.ABCD_F16,
                                     None, out, state)
        ab.abcd_backward(ctx, theta, cams[ci], None, proj, tiles, None, None, ab.ABCD_F16, None,
                         out, state, gt, 0.2, loss[k:k + 1], None, grads)
    step(0, pick[0])
    ctx.sync()
    Ks, lmean, lmax, walked, ms_all = [], [], [], [], []
    for k, ci in enumerate(pick):
        e0 = torch_event(torch, ctx.stream)
        step(k, ci)
        e1 = torch_event(torch, ctx.stream)
        ctx.sync()
        ms_all.append(e0.elapsed_time(e1))
        K = int(tiles.count.item())
        r = tiles.ranges.long()
        lens = (r[:, 1] - r[:, 0]).clamp(min=0)
        Ks.append(K)
        lmean.append(float(lens.double().mean()))
        lmax.append(int(lens.max()))
        walked.append(int(state.n_last.sum(dtype=torch.int64)))
    ms = float(np.mean(ms_all))
    res = {"workload": f"one block of {n} Gaussians (SH 3, 16-blob mixture), {width}x{height}, "
                       f"{len(pick)} of {n_cams} ring cameras",
           "fwd_bwd_steps_per_s": round(1e3 / ms, 2), "ms_per_step": round(ms, 3),
           "K_mean": int(np.mean(Ks)), "list_len_mean": round(float(np.mean(lmean)), 1),
           "list_len_max": int(np.max(lmax)), "pixel_list_pairs_walked_mean": int(np.mean(walked)),
           "pairs_per_s": round(float(np.mean(walked)) / (ms * 1e-3), 1)}
    del theta, grads, proj, tiles
    torch.cuda.empty_cache()
    return res


def run_medium_stage(device, T=100, seed=1002):
    """The 3x3x3 grid x 20,000 Gaussians (SH 3) workload, 50 hemisphere cameras at 640x480: one
    ABCD stage of the centre partition through the BCD driver (F/B composited from the cached
    layers of the visible pairs, T = 100 Adam steps, refresh), timed with events."""
    import torch
    import paper_2608_27735_gb300 as ab
    from paper_2608_27735_gb300 import scenegen as sg
    from paper_2608_27735_gb300.bcd import BCD, default_lr
    s = sg.medium_scene(seed=seed)
    tgt = sg.perturbed(s.gaussians, s.grid.side, seed=seed + 1)
    ref = BCD(tgt, (1, 1, 1), s.grid.origin, 3 * s.grid.side, s.cameras,
              np.zeros((len(s.cameras), 480, 640, 3), np.float32), 0, default_lr(15.0),
              max_pairs=40_000_000)
    targets = np.stack([ref.render_full(ci)[..., :3].cpu().numpy() for ci in range(len(s.cameras))])
    del ref
    run = BCD(s.gaussians, s.grid.dims, s.grid.origin, s.grid.side, s.cameras, targets, T,
              default_lr(15.0), seed=seed, max_pairs=8_000_000)
    centre = 13
    run.stage(centre)
    run.ctx.sync()
    e0 = torch_event(torch, run.ctx.stream)
    run.stage(centre)
    e1 = torch_event(torch, run.ctx.stream)
    run.ctx.sync()
    ms = e0.elapsed_time(e1)
    res = {"workload": "3x3x3 grid x 20000 Gaussians (SH 3), 50 hemisphere cameras 640x480, "
                       f"centre partition, T={T} steps per stage",
           "stage_ms": round(ms, 2), "active_steps_per_s": round(T / (ms * 1e-3), 1),
           "observing_cameras": len(run.cameras_of(centre)),
           "visible_pairs": int(run.frustum.sum()), "pairs": int(run.frustum.size),
           "loss_mean_first_last_10_steps": [round(float(run.loss[:10].mean()), 5),
                                             round(float(run.loss[T - 10:].mean()), 5)]}
    del run
    torch.cuda.empty_cache()
    return res


def run_visibility(st: Stage, reps=3):
    """Section 4's visibility threshold and occlusion culling on the stage's cache: every
    observing camera's layers (the active one as last refreshed) in its depth order, one
    abcd_layer_visibility_packed call per camera, timed on the context's stream; the pairs
    whose visible share is below TAU_VISIBLE, the stored bytes they hold and the bound on the
    composite error that dropping them gives.  The calls read every camera's stored tiles in
    turn (many GB, no L2 reuse)."""
    torch, ab = st.torch, st.ab
    P, a = st.n_parts, st.active
    cams = st.observing
    C = len(cams)
    vis = torch.empty(C, P, dtype=torch.float64, device=st.dev)
    cov = torch.empty_like(vis)
    tables = []
    for ci in cams:
        f, b = st.splits[ci]
        maps = [st.pk_map[ci, p] for p in range(P)]
        data = [st.pk_frozen[ci][st.pk_off[ci][p]:] if p != a else st.pk_active[ci] for p in range(P)]
        tables.append(ab.PackedLayers(maps, data, f + [a] + b, P))

    def sweep():
        for j in range(C):
            ab.abcd_layer_visibility_tables(st.ctx, tables[j], st.W, st.H, vis[j], cov[j])

    sweep()
    st.ctx.sync()
    e0 = torch_event(torch, st.stream)
    for _ in range(reps):
        sweep()
    e1 = torch_event(torch, st.stream)
    st.ctx.sync()
    us = e0.elapsed_time(e1) * 1e3 / (reps * C)
    v, c = vis.cpu().numpy(), cov.cpu().numpy()
    keep = ab.cull_pairs(v, c, TAU_VISIBLE)
    keep[:, a] = True                     # the active block's own pairs are being trained
    counts = st.pk_count.cpu().numpy()[cams].astype(np.int64)
    stored = int(counts.sum()) * 2048
    per_cam = stored / C + P * st.n_t * 4
    frozen = np.ones(P, bool)
    frozen[a] = False
    culled = (~keep) & frozen[None, :]
    culled_bytes = int(counts[culled].sum()) * 2048
    bound = float(np.where(culled, v, 0.0).sum(axis=1).max())
    peaks = load_peaks()
    peak = peaks["hbm_gbs"] if peaks else 6800.0
    gbs = per_cam / (us * 1e-6) / 1e9
    return {"tau_visible": TAU_VISIBLE, "pairs": C * (P - 1), "culled_pairs": int(culled.sum()),
            "frozen_cache_bytes": int(st.cache_bytes), "culled_bytes": culled_bytes,
            "max_mean_error_bound": round(bound, 6),
            "mean_visible_of_culled": round(float(v[culled].mean()), 7) if culled.any() else None,
            "us_per_camera": round(us, 2), "algorithmic_bytes_per_camera": int(per_cam),
            "gbs": round(gbs, 1), "hbm_frac": round(gbs / peak, 4),
            "kernel": "visibility_kernel<true>"}


def run_e2e(st: Stage, args, world, barrier):
    """The same stages with their inputs in pinned host memory (the host tier of the cache).
    Every stage, each observing camera's frozen layers (tile maps and stored tiles of the
    packed format) and target go host -> device on the context's copy stream
    (abcd_cache_fetch); a camera's copies for the next stage start as soon as this stage's
    composite of that camera has read its buffers (abcd_cache_release), so they overlap this
    stage's steps, as in the steady state of a training loop.  The refreshed layers go back on
    the other copy stream (abcd_cache_store); the parameters come in and go back, and the
    per-step losses go back, on the compute stream."""
    torch, ab = st.torch, st.ab
    C = len(st.cams)
    P, a = st.n_parts, st.active
    host_frozen = [t.cpu().pin_memory() for t in st.pk_frozen]
    host_maps = st.pk_map.cpu().pin_memory()
    host_gt = st.gt.cpu().pin_memory()
    theta_host = [t.cpu().pin_memory() for t in st.theta.tensors()]
    pool = min(8, C)
    refreshed = torch.empty(pool, st.n_t, 16, 16, 4, dtype=torch.float16, pin_memory=True)
    refreshed_map = torch.empty(pool, st.n_t, dtype=torch.int32, pin_memory=True)
    loss_host = torch.empty(args.T, dtype=torch.float32, pin_memory=True)
    gts = [st.gt, torch.empty_like(st.gt)]          # targets of this stage / the next one
    counted = {"h2d": 0, "d2h": 0}

    def fetch(ci, gt_dst):
        """Queues the host -> device copies of camera ci's inputs; returns their bytes."""
        n = 0
        for lo, hi in ((0, a), (a + 1, P)):
            if hi > lo:
                ab.abcd_cache_fetch(st.ctx, ci, host_maps[ci, lo:hi], st.pk_map[ci, lo:hi])
                n += (hi - lo) * st.n_t * 4
        ab.abcd_cache_fetch(st.ctx, ci, host_frozen[ci], st.pk_frozen[ci])
        n += host_frozen[ci].numel() * 2
        ab.abcd_cache_fetch(st.ctx, ci, host_gt[ci], gt_dst[ci])
        return n + host_gt[ci].numel() * 4

    def stage(k):
        cur, nxt = gts[k % 2], gts[(k + 1) % 2]
        h2d = d2h = 0
        for dst, src in zip(st.theta.tensors(), theta_host):
            dst.copy_(src, non_blocking=True)
            h2d += src.numel() * 4
        for x in (st.m, st.v):
            for tns in x.tensors():
                tns.zero_()
        for ci in st.observing:
            ab.abcd_cache_wait(st.ctx, ci)           # this stage's layers and target landed
            st.composite_one(ci)
            ab.abcd_cache_release(st.ctx, ci)
            h2d += fetch(ci, nxt)                     # the next stage's, behind this composite
        st.gt = cur
        for t in range(args.T):
            st.step(t, t)
        loss_host.copy_(st.loss, non_blocking=True)
        d2h += st.loss.numel() * 4
        st.refresh_all()
        for ci in st.observing:
            ab.abcd_cache_store(st.ctx, ci, st.pk_active[ci], refreshed[ci % pool])
            ab.abcd_cache_store(st.ctx, ci, st.pk_map[ci, a], refreshed_map[ci % pool])
            d2h += st.pk_active[ci].numel() * 2 + st.n_t * 4
        for src, dst in zip(st.theta.tensors(), theta_host):
            dst.copy_(src, non_blocking=True)
            d2h += src.numel() * 4
        counted.update(h2d=h2d, d2h=d2h)

    # the first stage's inputs, then one untimed stage that fetches the next one's
    for ci in st.observing:
        fetch(ci, gts[0])
    stage(0)
    torch.cuda.synchronize()
    st.sample_every = 10 ** 9
    barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    e0 = torch_event(torch, st.stream)
    h0 = time.perf_counter()
    for k in range(args.steps):
        stage(k + 1)
    host_ms = (time.perf_counter() - h0) * 1e3
    e1 = torch_event(torch, st.stream)
    ab.abcd_cache_sync(st.ctx)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    barrier()
    ms = max(e0.elapsed_time(e1), wall * 1e3)
    print(f"[bench] e2e: host issue time {host_ms / args.steps:.1f} ms, device {e0.elapsed_time(e1) / args.steps:.1f} ms, "
          f"wall {wall * 1e3 / args.steps:.1f} ms per stage", file=sys.stderr, flush=True)
    ms = max_over_ranks(ms, world)
    st.gt = gts[0]
    return {"value": round(args.steps * args.T * world / (ms / 1e3), 2), "unit": UNIT,
            "h2d_bytes_per_step": int(counted["h2d"]), "d2h_bytes_per_step": int(counted["d2h"]),
            "note": "per stage: active parameters, observing cameras' frozen layers (packed: tile "
                    "maps and stored tiles) and targets host->device (layers and targets on the "
                    "copy stream, one stage ahead); refreshed layers, parameters and losses "
                    "device->host"}


def run_streaming(st: Stage, args, world, barrier):
    """One F/B pair at a time (the host tier's streaming mode): no camera's layers, F, B or
    target stay on the device between steps.  For each step the sampled camera's frozen
    layers (packed) and target come from pinned host memory into one of two device slots,
    are composited into that slot's F/B pair, and the step runs; the next camera's copies are
    queued before the step, so they overlap it.  The refresh renders each camera's active
    layer into one of two device buffers and stores it back.  Device bytes for the cache, F,
    B and targets: two slots, whatever the number of cameras or partitions."""
    torch, ab = st.torch, st.ab
    P, a = st.n_parts, st.active
    host_frozen = [t.cpu().pin_memory() for t in st.pk_frozen]
    host_maps = st.pk_map.cpu().pin_memory()
    host_gt = st.gt.cpu().pin_memory()
    theta_host = [t.cpu().pin_memory() for t in st.theta.tensors()]
    loss_host = torch.empty(args.T, dtype=torch.float32, pin_memory=True)
    cap = max(t.shape[0] for t in st.pk_frozen)
    dev = st.dev
    slots = [dict(frozen=torch.empty(cap, 16, 16, 4, dtype=torch.float16, device=dev),
                  maps=torch.empty(P, st.n_t, dtype=torch.int32, device=dev),
                  gt=torch.empty(st.H, st.W, 3, device=dev),
                  F=torch.empty(st.H, st.W, 4, dtype=torch.float16, device=dev),
                  B=torch.empty(st.H, st.W, 4, dtype=torch.float16, device=dev)) for _ in range(2)]
    # refresh: each side context renders into its own two buffers and stores them back
    for w in st.side:
        w["active"] = [torch.empty(st.n_t, 16, 16, 4, dtype=torch.float16, device=dev) for _ in range(2)]
        w["back"] = [torch.empty(st.n_t, 16, 16, 4, dtype=torch.float16, pin_memory=True) for _ in range(2)]
        w["back_map"] = [torch.empty(st.n_t, dtype=torch.int32, pin_memory=True) for _ in range(2)]
        w["active_map"] = [torch.empty(st.n_t, dtype=torch.int32, device=dev) for _ in range(2)]
        w["active_cnt"] = torch.zeros(2, dtype=torch.int32, device=dev)
    dev_bytes = sum(sum(v.numel() * v.element_size() for v in s_.values()) for s_ in slots) + \
        sum(x.numel() * x.element_size() for w in st.side for x in w["active"] + w["active_map"])
    train = ab.TrainStep(st.ctx, st.theta, st.grads, st.m, st.v, st.proj, st.tiles, st.out,
                         st.state, LR)
    rng = np.random.default_rng(11)

    def fetch(k, ci):
        sl = slots[k]
        for lo, hi in ((0, a), (a + 1, P)):
            if hi > lo:
                ab.abcd_cache_fetch(st.ctx, k, host_maps[ci, lo:hi], sl["maps"][lo:hi])
        n = host_frozen[ci].shape[0]
        ab.abcd_cache_fetch(st.ctx, k, host_frozen[ci], sl["frozen"][:n])
        ab.abcd_cache_fetch(st.ctx, k, host_gt[ci], sl["gt"])

    def composite(k, ci):
        sl = slots[k]
        f, b = st.splits[ci]
        maps = [sl["maps"][p] if p != a else None for p in range(P)]
        data = [sl["frozen"][st.pk_off[ci][p]:] if p != a else None for p in range(P)]
        ab.abcd_composite_cache_packed(st.ctx, maps, data, f + [a] + b, len(f), st.W, st.H,
                                       sl["F"], sl["B"])

    def stage():
        for dst, src in zip(st.theta.tensors(), theta_host):
            dst.copy_(src, non_blocking=True)
        for x in (st.m, st.v):
            for tns in x.tensors():
                tns.zero_()
        order = []
        while len(order) < args.T:
            order += list(rng.permutation(st.observing))
        fetch(0, order[0])
        for t in range(args.T):
            k = t % 2
            ab.abcd_cache_wait(st.ctx, k)
            composite(k, order[t])
            if t + 1 < args.T:
                fetch(1 - k, order[t + 1])        # behind the step that last used that slot
            train(st.cams[order[t]], slots[k]["F"], slots[k]["B"], slots[k]["gt"],
                  st.loss[t:t + 1], t + 1)
            ab.abcd_cache_release(st.ctx, k)
        loss_host.copy_(st.loss, non_blocking=True)
        fork = torch_event(torch, st.stream)
        for w in st.side:
            w["ctx"].stream.wait_event(fork)
        nw = len(st.side)
        for j, ci in enumerate(st.observing):
            w = st.side[j % nw]
            k = (j // nw) % 2
            ab.abcd_cache_wait(w["ctx"], k)        # this buffer's previous store has left
            st.render_packed(st.theta, ci, w["active"][k], a, w, w["active_map"][k],
                             w["active_cnt"][k:k + 1])
            ab.abcd_cache_store(w["ctx"], k, w["active"][k], w["back"][k])
            ab.abcd_cache_store(w["ctx"], k, w["active_map"][k], w["back_map"][k])
        for w in st.side:
            st.stream.wait_event(torch_event(torch, w["ctx"].stream))
        for src, dst in zip(st.theta.tensors(), theta_host):
            dst.copy_(src, non_blocking=True)

    stage()
    torch.cuda.synchronize()
    st.sample_every = 10 ** 9
    barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    e0 = torch_event(torch, st.stream)
    for _ in range(args.steps):
        stage()
    e1 = torch_event(torch, st.stream)
    ab.abcd_cache_sync(st.ctx)
    for w in st.side:
        ab.abcd_cache_sync(w["ctx"])
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    barrier()
    ms = max(e0.elapsed_time(e1), wall * 1e3)
    ms = max_over_ranks(ms, world)
    per_step = sum(host_frozen[c].numel() * 2 + (P - 1) * st.n_t * 4 + host_gt[c].numel() * 4
                   for c in st.observing) / len(st.observing)
    return {"value": round(args.steps * args.T * world / (ms / 1e3), 2), "unit": UNIT,
            "device_bytes_cache_fb_targets": int(dev_bytes),
            "h2d_bytes_per_active_step": int(per_step),
            "note": "one F/B pair at a time: per step the sampled camera's packed frozen layers "
                    "and target are copied from pinned host memory (one step ahead) and "
                    "composited; the refresh stores each camera's layer back; the device holds "
                    "two slots whatever the number of cameras and partitions"}


# ---------------------------------------------------------------------------------------
# the oracle on the host cores (bounded sample of the same workload)

def oracle_sample(args, seed=1003):
    import oracle
    from paper_2608_27735_gb300 import scenegen as sg
    oracle.build()
    scene = sg.scene_scale(seed=seed, per_cell=args.per_cell, width=args.width,
                           height=args.height, n_cams=1)
    g = scene.gaussians
    cells = oracle.assign_cells(g.means, scene.grid.origin, scene.grid.side, scene.grid.dims)
    gx, gy, _ = scene.grid.dims
    active = ACTIVE_CELL[0] + gx * (ACTIVE_CELL[1] + gy * ACTIVE_CELL[2])
    ga = g.subset(np.nonzero(cells == active)[0])
    cam = scene.cameras[0]
    H, W = args.height, args.width
    L = sg.premultiplied_layers(2, H, W, seed=seed + 2).astype(np.float16).astype(np.float64)
    gt = sg.random_image(H, W, 3, seed=seed + 3).astype(np.float64)
    return oracle, ga, cam, L[0], L[1], gt


def oracle_step(oracle, ga, cam, F, B, gt, state):
    P = oracle.project(ga, cam)
    off, ids = oracle.tile_lists(P, cam.width, cam.height)
    sp = oracle.SplatSet.from_proj(P)
    R = oracle.render(sp, off, ids, cam.width, cam.height, F=F, B=B)
    L, dL = oracle.loss(R["out"][..., :3], gt, 0.2)
    g2 = oracle.backward(sp, off, ids, cam.width, cam.height, dL, F=F, B=B)
    gr = oracle.project_backward(ga, cam, g2)
    for k, name in enumerate(("means", "log_scales", "quats", "opacity_logits")):
        oracle.adam(state["theta"][k], gr[name], state["m"][k], state["v"][k], LR[k], 0.9, 0.999,
                    1e-15, state["step"])
    state["step"] += 1
    return L


def cpu_baseline(args, log):
    t0 = time.time()
    oracle, ga, cam, F, B, gt = oracle_sample(args)
    state = {"theta": [np.ascontiguousarray(a, dtype=np.float64) for a in ga.arrays()[:4]],
             "step": 1}
    state["m"] = [np.zeros_like(a) for a in state["theta"]]
    state["v"] = [np.zeros_like(a) for a in state["theta"]]
    log(f"[bench] oracle sample ready in {time.time() - t0:.1f}s")
    t1 = time.perf_counter()
    steps = 0
    while steps < 6 and (steps == 0 or time.perf_counter() - t1 < 10.0):
        oracle_step(oracle, ga, cam, F, B, gt, state)
        steps += 1
    dt = time.perf_counter() - t1
    return {"value": round(steps / dt, 5), "unit": UNIT, "cores": oracle.cpu_threads(),
            "kind": "oracle",
            "sample": f"{steps} active-block steps (project, bin/sort, render+composite, "
                      f"L1+D-SSIM, backward, Adam) of the same workload on one camera, "
                      f"{dt:.1f} s"}


def stage_config(args, n_active, world):
    """The workload both arms name (their JSON lines carry the same config)."""
    return {"workload": f"scene-scale ABCD stage: 4x4x2 grid x {args.per_cell} Gaussians/cell "
                        f"(SH3), {args.cams} cameras {args.width}x{args.height}, active cell "
                        f"{ACTIVE_CELL}, T={args.T} steps per stage, L1+0.2 D-SSIM",
            "bench_step": "one ABCD stage: composite F/B for the observing cameras (K1), "
                          "T active-block steps (K2-K9), cache refresh (K10)",
            "T": args.T, "observing_cameras": args.cams, "active_gaussians": int(n_active),
            "parallelism": f"replicas x{world}",
            "l2": "stage inputs exceed L2 (every stage reads all observing cameras' stored "
                  "layer tiles, many GB)"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    log = (lambda *a: print(*a, file=sys.stderr, flush=True))
    oracle, ga, cam, F, B, gt = oracle_sample(args)
    state = {"theta": [np.ascontiguousarray(a, dtype=np.float64) for a in ga.arrays()[:4]],
             "step": 1}
    state["m"] = [np.zeros_like(a) for a in state["theta"]]
    state["v"] = [np.zeros_like(a) for a in state["theta"]]
    for _ in range(args.warmup):
        oracle_step(oracle, ga, cam, F, B, gt, state)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(oracle, ga, cam, F, B, gt, state)
    dt = time.perf_counter() - t0
    v = args.steps / dt
    sample = (f"each timed step: one active-block step (K2-K9) of this workload on one camera "
              f"({ga.n} Gaussians, {args.width}x{args.height}); steps/s of the same unit as the "
              f"other arm's value")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(v, 5), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt * 1e3 / args.steps, 1),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": stage_config(args, ga.n, world),
        "cpu_baseline": {"value": round(v, 5), "unit": UNIT, "cores": oracle.cpu_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(v, 5), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
