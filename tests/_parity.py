"""Parity machinery: CUDA path (fp32) versus the fp64 oracle, element by element.

Where an fp32 computation decides something discrete (a radius, a tile boundary, whether a
Gaussian is skipped at a pixel, where a pixel's blend stops), both outcomes are correct when
the exact (fp64) value lies within fp32 rounding reach of the threshold.  This module derives
those ambiguous decisions from the oracle's own values with a stated uncertainty model, and
enumerates the oracle's result for every combination of them; the GPU must equal one of the
valid results (within the float tolerance) and everything else exactly.

Uncertainty model (u = 2^-24, unit roundoff of fp32):
  * camera-space mean:   dt_k = 8u (sum_j |R_kj mu_j| + |t_k|)
  * pixel-space mean:    du = fx (dt_x + |t_x/t_z| dt_z)/t_z + 8u (|fx t_x/t_z| + |cx|), same for v
  * conic (relative):    64u (1 + lambda_max/lambda_min)
  * radius (relative):   1e-5 on 3 sqrt(lambda_max)
  * sigma (relative, w.r.t. its absolute terms): 64u;   alpha: 4e-6;   transmittance step: 8u
"""
from __future__ import annotations

import itertools
import math

import numpy as np

import oracle

U = 2.0 ** -24
TOL_PIX = 1e-4
K_ARITH = 64 * U
EPS_ALPHA = 4e-6
EPS_STEP = 8 * U


def margins(g, cam, P):
    """Per-Gaussian absolute uncertainty of (u, v) and relative uncertainty of the conic."""
    R = np.asarray(cam.R, np.float64).reshape(3, 3)
    t = np.asarray(cam.t, np.float64)
    mu = np.asarray(g.means, np.float64)
    terms = np.abs(mu[:, None, :] * R[None, :, :]).sum(-1) + np.abs(t)[None, :]   # [n,3]
    dt = 8 * U * terms
    tc = mu @ R.T + t
    tz = np.where(np.abs(tc[:, 2]) > 1e-9, tc[:, 2], 1e-9)
    du = cam.fx * (dt[:, 0] + np.abs(tc[:, 0] / tz) * dt[:, 2]) / np.abs(tz) + \
        8 * U * (np.abs(cam.fx * tc[:, 0] / tz) + abs(cam.cx))
    dv = cam.fy * (dt[:, 1] + np.abs(tc[:, 1] / tz) * dt[:, 2]) / np.abs(tz) + \
        8 * U * (np.abs(cam.fy * tc[:, 1] / tz) + abs(cam.cy))
    lam = P["eig"]
    kappa = np.where(lam[:, 1] > 0, lam[:, 0] / np.maximum(lam[:, 1], 1e-30), 1.0)
    m_uv = np.stack([du, dv], -1)
    m_conic = 64 * U * (1 + kappa)
    return m_uv, m_conic


def splats_with_margins(g, cam, P):
    m_uv, m_c = margins(g, cam, P)
    return oracle.SplatSet.from_proj(P, m_uv=m_uv, m_conic=m_c, k_arith=K_ARITH,
                                     eps_alpha=EPS_ALPHA, eps_step=EPS_STEP)


def near_tiles(P, cam, m_uv, tiles, tile=16):
    """Gaussians whose tile rectangle, under any admissible fp32 rounding, may meet one of
    `tiles` (a superset: every other Gaussian is listed in none of them either way)."""
    tx, ty = oracle.tiles_xy(cam.width, cam.height, tile)
    ind = np.zeros((ty + 1, tx + 1), np.int64)
    for t in tiles:
        ind[t // tx + 1, t % tx + 1] = 1
    S = ind.cumsum(0).cumsum(1)
    r = np.ceil(P["radius_exact"] * (1 + 1e-5)) + 1
    u, v = P["uv"][:, 0], P["uv"][:, 1]
    cl = lambda a, m: np.clip(a, 0, m).astype(np.int64)
    x0 = cl(np.floor((u - m_uv[:, 0] - r) / tile), tx)
    x1 = cl(np.floor((u + m_uv[:, 0] + r) / tile) + 1, tx)
    y0 = cl(np.floor((v - m_uv[:, 1] - r) / tile), ty)
    y1 = cl(np.floor((v + m_uv[:, 1] + r) / tile) + 1, ty)
    cnt = S[y1, x1] - S[y0, x1] - S[y1, x0] + S[y0, x0]
    live = (P["depth"] > 0.2) & (P["radius_exact"] > 0)
    return np.nonzero(live & (cnt > 0))[0]


def rect_bounds(P, cam, m_uv, tile=16, idx=None):
    """Smallest and largest tile rectangle any admissible fp32 rounding can give (for the
    Gaussians idx only, all if None; the others get empty rectangles).  The candidates are
    the rectangles of both roundings of the radius (ceil of 3 sqrt(lambda_max) at its
    relative uncertainty) and of the corners of the (u, v) uncertainty box."""
    tx, ty = oracle.tiles_xy(cam.width, cam.height, tile)
    n = P["visible"].shape[0]
    lo = np.zeros((n, 4), np.int64)
    hi = np.zeros((n, 4), np.int64)
    amb_radius = np.zeros(n, bool)
    sel = np.arange(n) if idx is None else np.asarray(idx, np.int64)
    sel = sel[(P["depth"][sel] > 0.2) & (P["radius_exact"][sel] != 0)]
    if sel.size == 0:
        return lo, hi, amb_radius
    re = P["radius_exact"][sel].astype(np.float64)
    r_lo, r_hi = np.ceil(re * (1 - 1e-5)), np.ceil(re * (1 + 1e-5))
    amb_radius[sel] = r_lo != r_hi
    u, v = P["uv"][sel, 0].astype(np.float64), P["uv"][sel, 1].astype(np.float64)
    du, dv = m_uv[sel, 0], m_uv[sel, 1]
    cx0, cy0, cx1, cy1 = [], [], [], []
    for r in (r_lo, r_hi):
        for uu in (u - du, u + du):
            for vv in (v - dv, v + dv):
                cx0.append(np.clip(np.floor((uu - r) / tile), 0, tx))
                cy0.append(np.clip(np.floor((vv - r) / tile), 0, ty))
                cx1.append(np.clip(np.floor((uu + r) / tile) + 1, 0, tx))
                cy1.append(np.clip(np.floor((vv + r) / tile) + 1, 0, ty))
    cx0, cy0, cx1, cy1 = (np.stack(c).astype(np.int64) for c in (cx0, cy0, cx1, cy1))
    lo[sel] = np.stack([cx0.max(0), cy0.max(0), cx1.min(0), cy1.min(0)], 1)
    hi[sel] = np.stack([cx0.min(0), cy0.min(0), cx1.max(0), cy1.max(0)], 1)
    return lo, hi, amb_radius


def _in(rect, x, y):
    return rect[0] <= x < rect[2] and rect[1] <= y < rect[3]


LOG2E = 1.4426950408889634


def listing_ambiguity(P, lo, hi, cam, alpha_min=1.0 / 255.0, tile=16, tiles=None, m_uv=None):
    """Entries (Gaussian, tile) the GPU may list or not.

    Both sides list by the renderer's listing rule (R1b): tile t of Gaussian g's square is
    listed when m, the least sigma over t's pixel-centre box in log2 units, is at most
    lim = (thr (1 + LIST_REL) + LIST_ABS) (1 + LIST_REL), thr = log2(o / alpha_min).  The GPU
    decides it in fp32 (the x-extent of the ellipse sigma' <= lim over the tile row's band), so
    an entry is optional only when m lies within fp32 reach of lim:
      |m - lim| <= delta_g (lim + 1) + |grad m| |d uv| + lambda |d uv|^2 / 2,
    delta_g = 2 m_conic + 1e-5 (the conic's relative uncertainty of the model above and about
    170 roundings of the extent arithmetic), |grad m| <= sqrt(2 lambda m) at the box minimum,
    lambda the largest eigenvalue of the log2-scaled conic, d uv the mean's uncertainty; or when
    the tile's place in the square is itself ambiguous (lo / hi rectangles).
    Returns (opt_list, opt_render): tile -> set of ids whose listing may differ, and the subset
    where the Gaussian might still reach alpha_min at a pixel (render alternatives needed; the
    band around lim lies above thr, so only square-boundary entries can be in it).  tiles: only
    these tiles (all if None)."""
    tx, ty = oracle.tiles_xy(cam.width, cam.height, tile)
    opt_list, opt_render = {}, {}
    lam = P["eig"]
    kappa = np.where(lam[:, 1] > 0, lam[:, 0] / np.maximum(lam[:, 1], 1e-30), 1.0)
    m_conic = 64 * U * (1 + kappa)
    duv = np.hypot(m_uv[:, 0], m_uv[:, 1]) if m_uv is not None else np.full(len(kappa), 1e-4)

    def visit(g, x, y):
        o = P["opacity"][g]
        u, v = P["uv"][g]
        if not o >= alpha_min:
            return
        thr = math.log2(o / alpha_min)
        lim = (thr * (1 + oracle.LIST_REL) + oracle.LIST_ABS) * (1 + oracle.LIST_REL)
        a, b, c = P["conic"][g]
        qmax = LOG2E * 0.5 * (a + c + math.hypot(a - c, 2 * b))
        m = LOG2E * oracle.box_min_sigma(P["conic"][g], x * tile + 0.5 - u,
                                         x * tile + tile - 0.5 - u,
                                         y * tile + 0.5 - v, y * tile + tile - 0.5 - v)
        band = (2 * m_conic[g] + 1e-5) * (lim + 1) + math.sqrt(2 * qmax * max(m, 0.0)) * duv[g] + \
            0.5 * qmax * duv[g] ** 2
        in_sq_certain = _in(lo[g], x, y)
        keep_certain = m <= lim - band
        keep_possible = m <= lim + band
        if (in_sq_certain and keep_certain) or not keep_possible:
            return
        t = y * tx + x
        opt_list.setdefault(t, set()).add(int(g))
        if m <= thr + band:
            opt_render.setdefault(t, set()).add(int(g))

    live = np.any(hi != 0, axis=1) & (P["depth"] > 0.2)
    if tiles is None:
        for g in np.nonzero(live)[0]:
            for y in range(hi[g, 1], hi[g, 3]):
                for x in range(hi[g, 0], hi[g, 2]):
                    visit(g, x, y)
    else:
        for t in sorted(set(int(t) for t in tiles)):
            x, y = t % tx, t // tx
            cand = live & (hi[:, 0] <= x) & (x < hi[:, 2]) & (hi[:, 1] <= y) & (y < hi[:, 3])
            for g in np.nonzero(cand)[0]:
                visit(g, x, y)
    return opt_list, opt_render


def optional_share(opt_list, K):
    """Optional entries over the listed pairs, for the test output."""
    n = sum(len(v) for v in opt_list.values())
    return n, n / max(K, 1)


def check_tile_lists(gpu_ranges, gpu_ids, off, ids, P, opt, n_tiles, tiles=None):
    """GPU lists == oracle lists up to optional members, sorted by (fp32 depth, id); over the
    given tiles (all if None)."""
    keys = P["depth_key"].astype(np.int64)
    for t in (range(n_tiles) if tiles is None else tiles):
        s, e = int(gpu_ranges[t, 0]), int(gpu_ranges[t, 1])
        L = [int(v) for v in gpu_ids[s:e]] if e > s else []
        O = [int(v) for v in ids[off[t]:off[t + 1]]]
        o = opt.get(t, set())
        assert [g for g in L if g not in o] == [g for g in O if g not in o], f"tile {t}"
        assert set(L) <= set(O) | o, f"tile {t}: unexpected members"
        k = [(keys[g], g) for g in L]
        assert k == sorted(k), f"tile {t}: not sorted by (depth, id)"


def pixel_alternatives(sp, lst_full, labels, px, py, events, F, B, bg, opts, max_toggles=4):
    """All valid (render, list, event flips) of one pixel: every subset of its ambiguous
    decisions flipped.  labels[k] is "in" (certain member), "opt_in" / "opt_out" (optional
    member, present / absent in the oracle's nominal list)."""
    toggles = [("m", g) for g, m in zip(lst_full, labels) if m != "in"]
    toggles += [("e", ev) for ev in events]
    if len(toggles) > max_toggles:
        return None
    outs = []
    for k in range(len(toggles) + 1):
        for sub in itertools.combinations(toggles, k):
            mem_flip = {g for kind, g in sub if kind == "m"}
            ev_flip = [ev for kind, ev in sub if kind == "e"]
            lst = [g for g, m in zip(lst_full, labels)
                   if m == "in" or (m == "opt_in") != (g in mem_flip)]
            r = oracle.render_pixel(sp, lst, px, py, F=F, B=B, bg=bg, toggles=ev_flip, opts=opts)
            outs.append((r, lst, ev_flip))
    return outs


def reaches(P, g, px, py, alpha_min=1.0 / 255.0, delta=1e-4):
    """Whether Gaussian g might reach alpha_min at pixel (px, py) (exact value, with slack)."""
    o = P["opacity"][g]
    if o < alpha_min:
        return False
    u, v = P["uv"][g]
    a, b, c = P["conic"][g]
    dx, dy = px + 0.5 - u, py + 0.5 - v
    sig = 0.5 * (a * dx * dx + c * dy * dy) + b * dx * dy
    return sig <= math.log(o / alpha_min) * (1 + delta) + delta


def opt_pixel_mask(P, opt, cam, tile=16):
    """Pixels where an optional member of their tile might contribute."""
    tx, _ = oracle.tiles_xy(cam.width, cam.height, tile)
    mask = np.zeros((cam.height, cam.width), bool)
    for t, gs in opt.items():
        y0, x0 = (t // tx) * tile, (t % tx) * tile
        for py in range(y0, min(y0 + tile, cam.height)):
            for px in range(x0, min(x0 + tile, cam.width)):
                if any(reaches(P, g, px, py) for g in gs):
                    mask[py, px] = True
    return mask


def tile_candidates(t, off, ids, P, opt, px, py):
    """Oracle's list of tile t merged with the optional members that matter at (px, py),
    with membership labels."""
    O = [int(v) for v in ids[off[t]:off[t + 1]]]
    o = {g for g in opt.get(t, set()) if reaches(P, g, px, py)}
    allg = sorted(set(O) | o, key=lambda g: (int(P["depth_key"][g]), g))
    lab = []
    for g in allg:
        if g in o:
            lab.append("opt_in" if g in O else "opt_out")
        else:
            lab.append("in")
    return allg, lab


def compare_render(gpu_out, gpu_T, R, sp, off, ids, P, opt, cam, F=None, B=None, bg=None,
                   opts=None, tol=TOL_PIX, tile=16):
    """Returns the number of pixels resolved through alternatives; asserts parity."""
    H, W = cam.height, cam.width
    tx, _ = oracle.tiles_xy(W, H, tile)
    ref = R["out"]
    flagged = (R["n_ev"] > 0) | opt_pixel_mask(P, opt, cam, tile)
    ok = ~flagged
    err = np.abs(gpu_out[ok] - ref[ok]).max() if ok.any() else 0.0
    assert err <= tol, f"max |gpu - oracle| on unambiguous pixels = {err}"
    errT = np.abs(gpu_T[ok] - R["T_final"][ok]).max() if ok.any() else 0.0
    assert errT <= tol, f"max |T_gpu - T_oracle| = {errT}"
    n_alt = 0
    for py, px in zip(*np.nonzero(flagged)):
        t = (py // tile) * tx + (px // tile)
        allg, lab = tile_candidates(t, off, ids, P, opt, px, py)
        evs = [tuple(e) for e in R["ev"][py, px][:min(R["n_ev"][py, px], R["ev"].shape[2])]]
        Fp = None if F is None else F[py, px]
        Bp = None if B is None else B[py, px]
        alts = pixel_alternatives(sp, allg, lab, px, py, evs, Fp, Bp, bg, opts)
        assert alts is not None, f"pixel {(px, py)}: too many ambiguous decisions"
        best = min(np.abs(gpu_out[py, px] - a[0]["out"]).max() for a in alts)
        assert best <= tol, f"pixel {(px, py)} matches no valid alternative ({best})"
        n_alt += 1
    return n_alt


def grad_envelope(sp, off, ids, P, opt, R, cam, G, F=None, B=None, bg=None, opts=None, tile=16):
    """Per-Gaussian [lo, hi] offsets of grad2d over the alternatives of ambiguous pixels."""
    H, W = cam.height, cam.width
    tx, _ = oracle.tiles_xy(W, H, tile)
    n = sp.s.n
    lo = np.zeros((n, 9))
    hi = np.zeros((n, 9))
    flagged = (R["n_ev"] > 0) | opt_pixel_mask(P, opt, cam, tile)
    pix = list(zip(*np.nonzero(flagged)))
    for py, px in pix:
        t = (py // tile) * tx + (px // tile)
        allg, lab = tile_candidates(t, off, ids, P, opt, px, py)
        evs = [tuple(e) for e in R["ev"][py, px][:min(R["n_ev"][py, px], R["ev"].shape[2])]]
        Fp = None if F is None else F[py, px]
        Bp = None if B is None else B[py, px]
        alts = pixel_alternatives(sp, allg, lab, px, py, evs, Fp, Bp, bg, opts)
        assert alts is not None
        nominal_lst = [int(v) for v in ids[off[t]:off[t + 1]]]
        base = oracle.backward_pixel(sp, nominal_lst, px, py, G[py, px], F=Fp, B=Bp, bg=bg,
                                     opts=opts)
        deltas = []
        for _, lst, evf in alts:
            g = oracle.backward_pixel(sp, lst, px, py, G[py, px], F=Fp, B=Bp, bg=bg,
                                      toggles=evf, opts=opts)
            deltas.append(g - base)
        D = np.stack(deltas)
        lo += D.min(0)
        hi += D.max(0)
    return lo, hi, len(pix)


def assert_grad_close(gpu, ref, lo=None, hi=None, rtol=1e-3, atol=1e-5, what="grad"):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    if lo is None:
        lo = np.zeros_like(ref)
        hi = np.zeros_like(ref)
    tol = np.maximum(rtol * np.abs(ref), atol)
    below = gpu < ref + lo - tol
    above = gpu > ref + hi + tol
    bad = below | above
    if bad.any():
        idx = np.argwhere(bad)[:8]
        det = [(tuple(i), float(gpu[tuple(i)]), float(ref[tuple(i)])) for i in idx]
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} entries out of tolerance; "
                             f"first: {det}")
