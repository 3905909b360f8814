"""abcd_loss_static: the loss entry point that allocates nothing, for callers that cannot
allocate device memory (their host application owns every allocation, or they must not
allocate inside a latency-critical loop).  Checked through the C ABI against abcd_loss, the
workspace-backed entry point, and against the oracle, on two calls in a row (the shared static
scratch keeps the previous call's contents); with the gradient output left out; and as the
first call of a fresh process, where it looks up its scratch before anything else has run on
the device.  Collected last on purpose."""
import ctypes as C
import os
import subprocess
import sys

import numpy as np
import pytest

import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _static_fn():
    lib = ab.lib()
    f = lib.abcd_loss_static
    f.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_float, C.c_void_p,
                  C.c_void_p]
    f.restype = C.c_int
    return f


def _ptr(t):
    return C.c_void_p(t.data_ptr()) if t is not None else C.c_void_p(None)


def test_loss_static_matches_workspace_loss_and_oracle():
    torch = pytest.importorskip("torch")
    import oracle
    ab.build()
    f = _static_fn()
    ctx = ab.Context(0)
    stream = ctx.stream.cuda_stream
    for call, (H, W, lam) in enumerate([(150, 211, 0.2), (64, 96, 0.2)]):
        ctx.reserve(1, 1, H * W)
        xn = sg.random_image(H, W, 4, seed=40 + call)
        yn = sg.random_image(H, W, 3, seed=60 + call)
        x = torch.from_numpy(xn).cuda()
        y = torch.from_numpy(yn).cuda()
        l_ref = torch.zeros(1, device="cuda")
        g_ref = torch.empty(H, W, 3, device="cuda")
        ab.abcd_loss(ctx, x, y, W, H, lam, l_ref, g_ref)
        l_st = torch.full((1,), float("nan"), device="cuda")
        g_st = torch.full((H, W, 3), float("nan"), device="cuda")
        st = f(C.c_void_p(stream), _ptr(x), _ptr(y), W, H, lam, _ptr(l_st), _ptr(g_st))
        assert st == ab.ABCD_OK
        ctx.sync()
        a, b = l_st.item(), l_ref.item()
        assert abs(a - b) <= 1e-5 * abs(b), (call, a, b)
        gs, gr = g_st.cpu().numpy(), g_ref.cpu().numpy()
        assert np.all(np.abs(gs - gr) <= 1e-3 * np.abs(gr) + 1e-6 * np.abs(gr).max()), call
        # and against the oracle (fp64) on the fp32 inputs, at the loss tolerance
        L, G = oracle.loss(xn[..., :3].astype(np.float64), yn.astype(np.float64), lam)
        assert abs(a - L) <= 1e-5 * abs(L), (call, a, L)
        assert np.all(np.abs(gs - G) <= 1e-3 * np.abs(G) + 1e-5 * np.abs(G).max()), call
    # the gradient output is optional: the loss alone, equal to the workspace path's
    l_only = torch.full((1,), float("nan"), device="cuda")
    st = f(C.c_void_p(stream), _ptr(x), _ptr(y), W, H, lam, _ptr(l_only), C.c_void_p(None))
    assert st == ab.ABCD_OK
    torch.cuda.synchronize()
    assert abs(l_only.item() - l_ref.item()) <= 1e-5 * abs(l_ref.item())
    # sizes beyond the static scratch are rejected before any launch
    big = f(C.c_void_p(stream), _ptr(x), _ptr(y), 8192, 8192, 0.2, _ptr(l_st), _ptr(g_st))
    assert big == ab.ABCD_ERR_WORKSPACE


_FRESH = r"""
import ctypes as C, sys
import numpy as np, torch
sys.path.insert(0, sys.argv[1])
import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg
lib = ab.lib()
f = lib.abcd_loss_static
f.argtypes = [C.c_void_p] * 3 + [C.c_int, C.c_int, C.c_float, C.c_void_p, C.c_void_p]
f.restype = C.c_int
H, W = 70, 133
x = torch.from_numpy(sg.random_image(H, W, 4, seed=3)).cuda()
y = torch.from_numpy(sg.random_image(H, W, 3, seed=4)).cuda()
ls = torch.full((1,), float("nan"), device="cuda")
gs = torch.full((H, W, 3), float("nan"), device="cuda")
s = torch.cuda.current_stream().cuda_stream
# the static entry point first, before any other call of the library in this process
assert f(C.c_void_p(s), C.c_void_p(x.data_ptr()), C.c_void_p(y.data_ptr()), W, H, 0.2,
         C.c_void_p(ls.data_ptr()), C.c_void_p(gs.data_ptr())) == 0
torch.cuda.synchronize()
ctx = ab.Context(0)
ctx.reserve(1, 1, H * W)
lr = torch.zeros(1, device="cuda"); gr = torch.empty(H, W, 3, device="cuda")
ab.abcd_loss(ctx, x, y, W, H, 0.2, lr, gr)
ctx.sync()
assert abs(ls.item() - lr.item()) <= 1e-5 * abs(lr.item()), (ls.item(), lr.item())
g1, g2 = gs.cpu().numpy(), gr.cpu().numpy()
assert np.all(np.abs(g1 - g2) <= 1e-3 * np.abs(g2) + 1e-6 * np.abs(g2).max())
print("fresh ok", ls.item())
"""


def test_loss_static_first_call_of_a_fresh_process():
    pytest.importorskip("torch")
    ab.build()
    r = subprocess.run([sys.executable, "-c", _FRESH, ROOT], capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0 and "fresh ok" in r.stdout, r.stdout + r.stderr
