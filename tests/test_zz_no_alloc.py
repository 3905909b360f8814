"""abcd_loss_static: the loss entry point that allocates nothing, for callers that cannot
allocate device memory (their host application owns every allocation, or they must not
allocate inside a latency-critical loop).  Checked through the C ABI against abcd_loss, the
workspace-backed entry point, on two calls in a row (the shared static scratch keeps the
previous call's contents).  Collected last on purpose."""
import ctypes as C

import numpy as np
import pytest

import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg

pytestmark = pytest.mark.gpu


def test_loss_static_matches_workspace_loss():
    torch = pytest.importorskip("torch")
    ab.build()
    lib = ab.lib()
    f = lib.abcd_loss_static
    f.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_float, C.c_void_p,
                  C.c_void_p]
    f.restype = C.c_int
    ctx = ab.Context(0)
    stream = ctx.stream.cuda_stream
    for call, (H, W, lam) in enumerate([(150, 211, 0.2), (64, 96, 0.2)]):
        ctx.reserve(1, 1, H * W)
        x = torch.from_numpy(sg.random_image(H, W, 4, seed=40 + call)).cuda()
        y = torch.from_numpy(sg.random_image(H, W, 3, seed=60 + call)).cuda()
        l_ref = torch.zeros(1, device="cuda")
        g_ref = torch.empty(H, W, 3, device="cuda")
        ab.abcd_loss(ctx, x, y, W, H, lam, l_ref, g_ref)
        l_st = torch.full((1,), float("nan"), device="cuda")
        g_st = torch.full((H, W, 3), float("nan"), device="cuda")
        st = f(C.c_void_p(stream), C.c_void_p(x.data_ptr()), C.c_void_p(y.data_ptr()), W, H, lam,
               C.c_void_p(l_st.data_ptr()), C.c_void_p(g_st.data_ptr()))
        assert st == ab.ABCD_OK
        ctx.sync()
        a, b = l_st.item(), l_ref.item()
        assert abs(a - b) <= 1e-5 * abs(b), (call, a, b)
        gs, gr = g_st.cpu().numpy(), g_ref.cpu().numpy()
        assert np.all(np.abs(gs - gr) <= 1e-3 * np.abs(gr) + 1e-6 * np.abs(gr).max()), call
    # sizes beyond the static scratch are rejected before any launch
    big = f(C.c_void_p(stream), C.c_void_p(x.data_ptr()), C.c_void_p(y.data_ptr()), 8192, 8192,
            0.2, C.c_void_p(l_st.data_ptr()), C.c_void_p(g_st.data_ptr()))
    assert big == ab.ABCD_ERR_WORKSPACE
