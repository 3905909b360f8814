"""A whole ABCD stage (Section 2) on the GPU against the oracle.

One stage of the tiny workload (2x2x2 grid x 2,000 Gaussians, SH 0, four 128x128 cameras on a
ring, L1 + 0.2 D-SSIM against targets rendered from a perturbed copy of the scene): the cached
renders of the frozen blocks composited into F and B, T = 10 Adam steps on the active block
with the cameras the driver samples, then the refresh of the block's cached renders.  Checked:

* the initial cache (every block's render for every camera, fp16) and F, B (the fold of the
  frozen layers in each camera's depth order, fp16) against the oracle's;
* every step along the stage's own trajectory: at the parameters the GPU held before the step,
  its loss and its gradient against the oracle's (loss 1e-5 relative; gradients element-wise at
  1e-3 relative / 1e-5 absolute, or in relative L2 norm at steps where a pixel has a decision
  within fp32 rounding of its threshold), and its Adam update against the oracle's Adam applied
  to the GPU's gradient (fp32 rounding);
* an independent fp64 oracle stage from the same start (its own cache, F, B, gradients and
  Adam, the same cameras): its losses against the GPU's at every step, and the parameters
  after the stage element-wise within the gradient tolerance carried through the T Adam
  updates (derivation in test_stage_matches_oracle);
* the refreshed layers against the oracle's render of the parameters the stage ended with;
* every frozen block's parameters and cached layers bit-identical after the stage.
"""
import numpy as np
import pytest

import oracle
import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg
from paper_2608_27735_gb300.bcd import BCD, default_lr
from tests import _parity as par

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

GROUPS = ("means", "log_scales", "quats", "opacity_logits", "sh")
T_STAGE = 10
LAM = 0.2
# the optimiser's hyperparameters as the C ABI receives them (fp32): (1 - beta2) in fp32 is
# 1.3e-5 away from 0.001, which the oracle must see too
BETA1, BETA2, EPS = float(np.float32(0.9)), float(np.float32(0.999)), float(np.float32(1e-15))


def host_gaussians(th):
    """scenegen.Gaussians (float32 numpy) from a block's device tensors."""
    a = [t.detach().cpu().numpy().copy() for t in th.tensors()]
    return sg.Gaussians(*a, th.sh_degree)


def oracle_render(g, cam, F=None, B=None):
    P = oracle.project(g, cam)
    off, ids = oracle.tile_lists(P, cam.width, cam.height)
    sp = par.splats_with_margins(g, cam, P)
    R = oracle.render(sp, off, ids, cam.width, cam.height, F=F, B=B)
    return P, off, ids, sp, R


def ambiguous(g, cam, P, R):
    """Whether any decision of this render lies within fp32 reach of its threshold."""
    m_uv, _ = par.margins(g, cam, P)
    lo, hi, amb_r = par.rect_bounds(P, cam, m_uv)
    _, opt = par.listing_ambiguity(P, lo, hi, cam, m_uv=m_uv)
    return bool((R["n_ev"] > 0).any() or opt or amb_r.any()), opt, P


def refresh_ok(got16, g, cam):
    """fp16 layer of block g for camera cam against the oracle: the RNE rounding of the exact
    value, except where the exact value is within 1e-4 (the fp32 pixel tolerance) of an fp16
    midpoint; pixels with an ambiguous decision are left out (returns their share)."""
    P, off, ids, sp, R = oracle_render(g, cam)
    _, opt, _ = ambiguous(g, cam, P, R)
    ok = (R["n_ev"] == 0) & ~par.opt_pixel_mask(P, opt, cam)
    ref = R["A"]
    lo, hi = (ref - 1e-4).astype(np.float16), (ref + 1e-4).astype(np.float16)
    gg = got16.astype(np.float64)
    assert np.all((gg[ok] >= lo[ok].astype(np.float64)) & (gg[ok] <= hi[ok].astype(np.float64)))
    exact = ok[..., None] & (lo == hi)
    assert np.all(got16[exact] == ref.astype(np.float16)[exact])
    return 1.0 - float(ok.mean())


def fb16_ok(got16, ref64, L):
    """fp16 fold output against the exact fold of the same fp16 layers (fp32 accumulation,
    one rounding: within the accumulated rounding L * 4u of the exact value)."""
    m = L * 4 * 2.0 ** -24 * np.abs(ref64)
    lo, hi = (ref64 - m).astype(np.float16), (ref64 + m).astype(np.float16)
    assert np.all((got16 >= lo) & (got16 <= hi))
    exact = lo == hi
    assert np.all(got16[exact] == ref64.astype(np.float16)[exact])


def masked_gradients(run, g, ci, cam, F64, B64, target, P, off, ids, sp, R, opt):
    """Both gradients of a step with the upstream gradient zeroed within 10 pixels (the reach of
    the SSIM windows' coupling) of every pixel that has a decision within fp32 rounding of its
    threshold: no such pixel then feeds either side, so they are compared element-wise.  The GPU
    side re-runs the step's kernels at the same parameters, camera, F and B.  Returns (GPU
    gradient groups, oracle gradient groups, share of pixels kept)."""
    from scipy import ndimage
    W, H = cam.width, cam.height
    bad = (R["n_ev"] > 0) | par.opt_pixel_mask(P, opt, cam)
    keep = ~ndimage.binary_dilation(bad, structure=np.ones((21, 21), bool))
    L, dL = oracle.loss(R["out"][..., :3], target.astype(np.float64), LAM)
    g2 = oracle.backward(sp, off, ids, W, H, dL * keep[..., None], F=F64, B=B64)
    ref = oracle.project_backward(g, cam, g2)
    c = run.cams[ci]
    th = ab.Gaussians.from_numpy(g)
    ab.abcd_project(run.ctx, th, c, None, run.proj)
    ab.abcd_bin_sort(run.ctx, run.proj, th.n, c, run.tiles)
    Ft = torch.from_numpy(F64.astype(np.float16)).cuda()
    Bt = torch.from_numpy(B64.astype(np.float16)).cuda()
    out = torch.empty(H, W, 4, device="cuda")
    state = ab.FwdState.alloc(W, H)
    ab.abcd_render_composite_fwd(run.ctx, c, None, run.proj, run.tiles, Ft, Bt, ab.ABCD_F16, None,
                                 out, state)
    loss = torch.zeros(1, device="cuda")
    dl = torch.empty(H, W, 3, device="cuda")
    ab.abcd_loss(run.ctx, out, torch.from_numpy(target).cuda(), W, H, LAM, loss, dl)
    dl *= torch.from_numpy(keep.astype(np.float32)).cuda()[..., None]
    grad2d = torch.empty(th.n, 9, device="cuda")
    ab.abcd_render_backward(run.ctx, c, None, run.proj, run.tiles, Ft, Bt, ab.ABCD_F16, None, state,
                            dl, th.n, grad2d)
    grads = ab.Gaussians.zeros_like(th)
    ab.abcd_project_backward(run.ctx, th, c, None, grad2d, grads)
    run.ctx.sync()
    return [t.cpu().numpy().astype(np.float64) for t in grads.tensors()], ref, float(keep.mean())


def oracle_adam(theta, grad, m, v, lr, step):
    """fp64 Adam on numpy group arrays (lists of 5), in place; SH degree 0 and the higher
    degrees take their own learning rates."""
    for k in range(5):
        if k < 4:
            oracle.adam(theta[k], grad[k], m[k], v[k], lr[k], BETA1, BETA2, EPS, step)
        else:
            for sl, l in ((np.s_[:, :1, :], lr[4]), (np.s_[:, 1:, :], lr[5])):
                if theta[4][sl].size == 0:
                    continue
                a, mm, vv = (np.ascontiguousarray(x[sl]) for x in (theta[4], m[4], v[4]))
                oracle.adam(a, np.ascontiguousarray(grad[k][sl]), mm, vv, l, BETA1, BETA2, EPS, step)
                theta[4][sl], m[4][sl], v[4][sl] = a, mm, vv


def group_lr(lr, k, shape):
    if k < 4:
        return np.full(shape, lr[k])
    out = np.full(shape, lr[5])
    out[:, :1, :] = lr[4]
    return out


def check_steps(run, rec, theta0, halo, cams, F64, B64, targets, lr, min_kept=0.3):
    """Every recorded step of a stage against the oracle at the parameters the GPU held before
    it: the loss, the gradient of the trained rows (element-wise, or with the pixels near an
    ambiguous decision left out of both sides plus in relative L2 norm) and the Adam update.
    halo: frozen Gaussians rendered after the trained ones (scenegen.Gaussians) or None;
    min_kept: the least share of pixels an ambiguous step may keep for its element-wise check."""
    W, H = cams[0].width, cams[0].height
    n = theta0.n
    th = [a.astype(np.float64) for a in theta0.arrays()]
    m_prev = [np.zeros_like(a) for a in th]
    v_prev = [np.zeros_like(a) for a in th]
    strict_steps = 0
    kept_share = []
    for t, r in enumerate(rec):
        ci = r["ci"]
        cam = cams[ci]
        parts = [a.astype(np.float32) for a in th]
        if halo is not None:
            parts = [np.concatenate([a, h]) for a, h in zip(parts, halo.arrays())]
        g = sg.Gaussians(*parts, theta0.sh_degree)
        P, off, ids, sp, R = oracle_render(g, cam, F64[ci], B64[ci])
        L, dL = oracle.loss(R["out"][..., :3], targets[ci].astype(np.float64), LAM)
        g2 = oracle.backward(sp, off, ids, W, H, dL, F=F64[ci], B=B64[ci])
        ref = {k: v[:n] for k, v in oracle.project_backward(g, cam, g2).items()}
        amb, opt, _ = ambiguous(g, cam, P, R)
        assert abs(r["loss"] - L) <= 1e-5 * L, (t, r["loss"], L)
        if amb:
            gm, refm, kept = masked_gradients(run, g, ci, cam, F64[ci], B64[ci], targets[ci], P, off,
                                              ids, sp, R, opt)
            gm = [x[:n] for x in gm]
            refm = {k: v[:n] for k, v in refm.items()}
            assert kept > min_kept, (t, kept)
            kept_share.append(kept)
        for k, name in enumerate(GROUPS):
            got = r["grad"][k].astype(np.float64)
            if not amb:
                atol = min(1e-5, 1e-5 * float(np.abs(ref[name]).max()))
                par.assert_grad_close(got, ref[name], rtol=1e-3, atol=atol, what=f"step {t} {name}")
            else:
                rel = np.linalg.norm(got - ref[name]) / max(np.linalg.norm(ref[name]), 1e-30)
                assert rel < 1e-3, (t, name, rel)
                atol = min(1e-5, 1e-5 * float(np.abs(refm[name]).max()))
                par.assert_grad_close(gm[k], refm[name], rtol=1e-3, atol=atol,
                                      what=f"step {t} {name} (unambiguous pixels)")
        strict_steps += not amb
        # the update: the oracle's Adam on the GPU's gradient from the GPU's state
        a, mm, vv = [x.copy() for x in th], [x.copy() for x in m_prev], [x.copy() for x in v_prev]
        oracle_adam(a, [x.astype(np.float64) for x in r["grad"]], mm, vv, lr, t + 1)
        for k in range(5):
            # m = b1 m + (1 - b1) g takes three fp32 roundings (two products, the sum), each at
            # most 2^-24 of the value it rounds: where the two terms nearly cancel, the error is
            # bounded by the terms, not by the (small) result
            g64 = r["grad"][k].astype(np.float64)
            terms = BETA1 * np.abs(m_prev[k].astype(np.float64)) + (1.0 - BETA1) * np.abs(g64)
            err_m = np.abs(r["m"][k].astype(np.float64) - mm[k])
            assert np.all(err_m <= 2e-6 * np.abs(mm[k]) + 3.0 * 2.0 ** -24 * terms + 1e-30), \
                (t, k, float(np.max(err_m - 2e-6 * np.abs(mm[k]) - 3.0 * 2.0 ** -24 * terms)))
            np.testing.assert_allclose(r["v"][k], vv[k], rtol=4e-6, atol=1e-18)
            np.testing.assert_allclose(r["theta"][k], a[k], rtol=2e-6, atol=2e-7)
        th, m_prev, v_prev = r["theta"], r["m"], r["v"]
    print(f"stage: {strict_steps} of {len(rec)} steps free of ambiguous decisions (whole gradient "
          f"element-wise); the others element-wise on the pixels kept ({np.mean(kept_share or [1]):.0%}"
          f" on average) and in relative L2 norm on all")


def recorder(rec):
    def trace(t, ci, th, grads, m, v, loss):
        rec.append(dict(ci=ci, theta=[x.cpu().numpy().astype(np.float64) for x in th.tensors()],
                        grad=[x.cpu().numpy() for x in grads.tensors()],
                        m=[x.cpu().numpy().astype(np.float64) for x in m.tensors()],
                        v=[x.cpu().numpy().astype(np.float64) for x in v.tensors()],
                        loss=float(loss.item())))
    return trace


def test_stage_matches_oracle():
    scene = sg.tiny_scene()
    dims, side, origin = scene.grid.dims, scene.grid.side, scene.grid.origin
    cams = scene.cameras
    W, H = cams[0].width, cams[0].height
    tgt = sg.perturbed(scene.gaussians, side, seed=2002)
    targets = []
    for cam in cams:
        Pt = oracle.project(tgt, cam)
        ot, it = oracle.tile_lists(Pt, W, H)
        targets.append(oracle.render(oracle.SplatSet.from_proj(Pt), ot, it, W, H)["out"][..., :3])
    targets = np.stack(targets).astype(np.float32)
    lr = [float(np.float32(x)) for x in default_lr(2 * side)]
    active = 0
    run = BCD(scene.gaussians, dims, origin, side, cams, targets, T_STAGE, lr, mode="abcd",
              seed=7, lambda_ssim=LAM)
    n_blocks = int(np.prod(dims))
    blocks = {b: scene.gaussians.subset(run.members[b]) for b in run.blocks}

    # ---- the initial cache: every block's render for every camera
    layers0 = run.layers.cpu().numpy()
    left_out = [refresh_ok(layers0[ci, b], blocks[b], cams[ci])
                for ci in range(len(cams)) for b in run.blocks]
    assert max(left_out) < 0.05, left_out

    frozen_theta = {b: [t.cpu().clone() for t in run.theta[b].tensors()]
                    for b in run.blocks if b != active}
    frozen_layers = run.layers[:, [b for b in range(n_blocks) if b != active]].cpu().clone()
    theta0 = host_gaussians(run.theta[active])

    rec = []

    def trace(t, ci, th, grads, m, v, loss):
        rec.append(dict(ci=ci, theta=[x.cpu().numpy().astype(np.float64) for x in th.tensors()],
                        grad=[x.cpu().numpy() for x in grads.tensors()],
                        m=[x.cpu().numpy().astype(np.float64) for x in m.tensors()],
                        v=[x.cpu().numpy().astype(np.float64) for x in v.tensors()],
                        loss=float(loss.item())))

    run.stage(active, trace=trace)
    run.ctx.sync()
    assert len(rec) == T_STAGE

    # ---- F and B of the stage: the fold of the frozen layers in each camera's order
    F16, B16 = run.F.cpu().numpy(), run.B.cpu().numpy()
    F64, B64 = {}, {}
    for ci in range(len(cams)):
        order, split = run.order[ci, active]
        front, back = order[:split], order[split + 1:]
        for lst, got, dst in ((front, F16, F64), (back, B16, B64)):
            if lst:
                ref = oracle.composite_layers(layers0[ci].astype(np.float64), list(lst))
            else:
                ref = np.zeros((H, W, 4))
            fb16_ok(got[ci], ref, max(1, len(lst)))
            dst[ci] = got[ci].astype(np.float64)

    # ---- every step at the GPU's own parameters
    check_steps(run, rec, theta0, None, cams, F64, B64, targets, lr)

    # ---- the refresh: the block's layers rendered from the parameters the stage ended with
    thetaT = host_gaussians(run.theta[active])
    layersT = run.layers.cpu().numpy()
    left_out = [refresh_ok(layersT[ci, active], thetaT, cams[ci]) for ci in range(len(cams))]
    assert max(left_out) < 0.05, left_out

    # ---- frozen blocks untouched, bit for bit
    for b, ts in frozen_theta.items():
        for a_, b_ in zip(ts, run.theta[b].tensors()):
            assert torch.equal(a_, b_.cpu()), b
    assert torch.equal(frozen_layers, run.layers[:, [b for b in range(n_blocks) if b != active]].cpu())

    # ---- an independent fp64 oracle stage from the same start
    Fo, Bo = {}, {}
    for ci in range(len(cams)):
        lay = {b: oracle_render(blocks[b], cams[ci])[4]["A"].astype(np.float16).astype(np.float64)
               for b in run.blocks if b != active}
        order, split = run.order[ci, active]
        for lst, dst in ((order[:split], Fo), (order[split + 1:], Bo)):
            if lst:
                keys = list(lst)
                st = np.stack([lay[k] for k in keys])
                dst[ci] = oracle.composite_layers(st, list(range(len(keys)))).astype(np.float16).astype(np.float64)
            else:
                dst[ci] = np.zeros((H, W, 4))
    tho = [a.astype(np.float64) for a in theta0.arrays()]
    mo = [np.zeros_like(a) for a in tho]
    vo = [np.zeros_like(a) for a in tho]
    # per element, the bound on how far the GPU's parameters may drift from the oracle's: each
    # step's gradient may differ by the benchmark spec's tolerance tau = 1e-3 |g| + 1e-5 max|g| (the
    # absolute floor per group); Adam's step lr * mhat / (sqrt(vhat) + eps) then differs, to
    # first order, by lr (|dm| / sqrt(vhat) + |mhat| |dv| / (2 vhat^1.5)) <= 3 lr tau / sqrt(vhat)
    # (the second term is at most 1.25 times the first, |mhat| / sqrt(vhat) <= 1.25 for the
    # first ten steps at these betas), and by at most 2 * 1.25 lr where the gradient is below
    # the floor (its sign is not fixed)
    drift = [np.zeros_like(a) for a in tho]
    max_loss_rel = 0.0
    for t, r in enumerate(rec):
        ci = r["ci"]
        cam = cams[ci]
        g = sg.Gaussians(*[a.astype(np.float32) for a in tho], theta0.sh_degree)
        P, off, ids, sp, R = oracle_render(g, cam, Fo[ci], Bo[ci])
        L, dL = oracle.loss(R["out"][..., :3], targets[ci].astype(np.float64), LAM)
        g2 = oracle.backward(sp, off, ids, W, H, dL, F=Fo[ci], B=Bo[ci])
        ref = oracle.project_backward(g, cam, g2)
        max_loss_rel = max(max_loss_rel, abs(r["loss"] - L) / L)
        gr = [ref[n] for n in GROUPS]
        oracle_adam(tho, gr, mo, vo, lr, t + 1)
        for k in range(5):
            floor = 1e-5 * float(np.abs(gr[k]).max())
            tau = 1e-3 * np.abs(gr[k]) + floor
            vhat = vo[k] / (1 - BETA2 ** (t + 1))
            step_tol = group_lr(lr, k, tho[k].shape) * np.where(
                np.abs(gr[k]) > floor, np.minimum(2.5, 3.0 * tau / np.maximum(np.sqrt(vhat), 1e-300)), 2.5)
            drift[k] += step_tol
    assert max_loss_rel <= 1e-4, max_loss_rel
    worst = 0.0
    for k, name in enumerate(GROUPS):
        got = run.theta[active].tensors()[k].cpu().numpy().astype(np.float64)
        d = np.abs(got - tho[k])
        tol = drift[k] + 1e-6 * np.abs(tho[k]) + 1e-7
        assert np.all(d <= tol), (name, float((d - tol).max()), int((d > tol).sum()))
        moved = np.abs(tho[k] - theta0.arrays()[k].astype(np.float64))
        worst = max(worst, float((d / np.maximum(moved, 1e-12))[moved > 1e-6].max(initial=0.0)))
    print(f"independent oracle stage: losses within {max_loss_rel:.2e} relative; parameters "
          f"within {worst:.2e} of their movement over the stage")


def test_overlap_stage_matches_oracle():
    """A stage with an overlapping boundary region (reading R17): block 0 of a 2x1x1 grid is
    trained together with its halo (block 1's Gaussians within 1.0 of its cell, rendered in the
    same depth sort, frozen), against F and B folded from block 1's layer re-rendered without
    them.  Checked against the oracle: the re-rendered donor layers, F and B as the fold of the
    layers the stage uses, every step (loss, the block's gradient, Adam on the block's rows
    only) at the parameters the GPU held, the block's refreshed layers, and the donor block
    bit-identical afterwards."""
    s = sg.grid_scene((2, 1, 1), 5.0, 300, 0, seed=11)
    g = s.gaussians
    cams = sg.ring_cameras(4, 1.5 * sg.half_diagonal(s.grid), np.zeros(3), 160, 120, seed=11)
    W, H = 160, 120
    tgt = sg.perturbed(g, 5.0, seed=12)
    targets = []
    for cam in cams:
        Pt = oracle.project(tgt, cam)
        ot, it = oracle.tile_lists(Pt, W, H)
        targets.append(oracle.render(oracle.SplatSet.from_proj(Pt), ot, it, W, H)["out"][..., :3])
    targets = np.stack(targets).astype(np.float32)
    lr = [float(np.float32(x)) for x in default_lr(10.0)]
    run = BCD(g, (2, 1, 1), s.grid.origin, 5.0, cams, targets, 6, lr, seed=4, lambda_ssim=LAM,
              overlap=1.0)
    b, q = 0, 1
    pos = run.halo[b][q]
    assert len(pos) > 10
    donor = host_gaussians(run.theta[q])
    halo = donor.subset(pos)
    core = donor.subset(np.setdiff1d(np.arange(donor.n), pos))
    theta0 = host_gaussians(run.theta[b])
    donor_before = [t.cpu().clone() for t in run.theta[q].tensors()]
    # the donor's layer without its halo members, as the stage's composite takes it
    cores = torch.empty(len(cams), H, W, 4, dtype=torch.float16, device="cuda")
    for ci in range(len(cams)):
        run._core_layer(q, pos, ci, cores[ci])
    run.ctx.sync()
    cores_np = cores.cpu().numpy()
    left_out = [refresh_ok(cores_np[ci], core, cams[ci]) for ci in range(len(cams))]
    assert max(left_out) < 0.05, left_out
    rec = []
    run.stage(b, trace=recorder(rec))
    run.ctx.sync()
    assert len(rec) == 6
    F16, B16 = run.F.cpu().numpy(), run.B.cpu().numpy()
    F64, B64 = {}, {}
    for ci in range(len(cams)):
        order, split = run.order[ci, b]
        for lst, got, dst in ((order[:split], F16, F64), (order[split + 1:], B16, B64)):
            if lst:
                assert list(lst) == [q]
                fb16_ok(got[ci], cores_np[ci].astype(np.float64), 1)
            else:
                assert not np.any(got[ci])
            dst[ci] = got[ci].astype(np.float64)
    check_steps(run, rec, theta0, halo, cams, F64, B64, targets, lr, min_kept=0.2)
    thetaT = host_gaussians(run.theta[b])
    layersT = run.layers.cpu().numpy()
    left_out = [refresh_ok(layersT[ci, b], thetaT, cams[ci]) for ci in range(len(cams))]
    assert max(left_out) < 0.05, left_out
    for a_, b_ in zip(donor_before, run.theta[q].tensors()):
        assert torch.equal(a_, b_.cpu())
