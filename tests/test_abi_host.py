"""Host-side checks of the C ABI (no GPU): the library loads, exports every function the
header declares, the ctypes mirrors match the C struct layouts, and the host partition
logic agrees with the oracle."""
import ctypes as C
import os
import subprocess

import numpy as np
import pytest

import oracle
import paper_2608_27735_gb300 as ab
from paper_2608_27735_gb300 import scenegen as sg


@pytest.fixture(scope="module")
def lib():
    ab.build()
    return ab.lib()


def test_exports_every_declared_function(lib):
    names = ab.header_functions()
    assert len(names) >= 20
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    for n in ("abcd_project", "abcd_bin_sort", "abcd_render_composite_fwd", "abcd_backward",
              "abcd_composite_cache", "abcd_adam_active"):
        assert n in names


def test_struct_layouts_match_header(tmp_path):
    src = tmp_path / "layout.c"
    structs = {"abcd_camera": ab.abcd_camera, "abcd_render_opts": ab.abcd_render_opts,
               "abcd_gaussians": ab.abcd_gaussians, "abcd_projected": ab.abcd_projected,
               "abcd_tiles": ab.abcd_tiles, "abcd_fwd_state": ab.abcd_fwd_state}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "abcd.h"', "int main(void){"]
    for name, py in structs.items():
        lines.append(f'printf("{name} %zu\\n", sizeof({name}));')
        for f, _ in py._fields_:
            lines.append(f'printf("{name}.{f} %zu\\n", offsetof({name}, {f}));')
    lines.append("return 0;}")
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(ab.HEADER))
    subprocess.run(["gcc", "-I", inc, str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    got = dict(l.rsplit(" ", 1) for l in out.strip().splitlines())
    for name, py in structs.items():
        assert int(got[name]) == C.sizeof(py), name
        for f, _ in py._fields_:
            assert int(got[f"{name}.{f}"]) == getattr(py, f).offset, (name, f)


def test_workspace_size(lib):
    sz = C.c_size_t()
    assert lib.abcd_workspace_size(1000, 10000, 4096, C.byref(sz)) == 0
    small = sz.value
    assert lib.abcd_workspace_size(2000, 10000, 4096, C.byref(sz)) == 0
    assert sz.value > small
    assert lib.abcd_workspace_size(-1, 0, 0, C.byref(sz)) == ab.ABCD_ERR_INVALID_ARG


def test_host_partition_logic_matches_oracle(lib):
    rng = np.random.default_rng(3)
    for trial in range(40):
        dims = tuple(int(v) for v in rng.integers(1, 5, 3))
        side = float(rng.uniform(0.5, 6))
        origin = rng.uniform(-10, 10, 3)
        campos = origin + rng.uniform(-2, np.array(dims) * side + 2)
        active = int(rng.integers(0, np.prod(dims)))
        f1, b1 = ab.abcd_partition_split(dims, origin, side, campos, active)
        f2, b2 = oracle.partition_split(dims, origin, side, campos, active)
        assert list(f1) == list(f2) and list(b1) == list(b2)
    s = sg.tiny_scene(per_cell=300)
    c1 = ab.abcd_assign_cells(s.gaussians.means, s.grid.origin, s.grid.side, s.grid.dims)
    c2 = oracle.assign_cells(s.gaussians.means, s.grid.origin, s.grid.side, s.grid.dims)
    np.testing.assert_array_equal(c1, c2)
    with pytest.raises(ab.AbcdError):
        ab.abcd_partition_split((2, 2, 2), (0, 0, 0), 1.0, (0, 0, 0), 8)


def test_no_cpu_fallback_without_gpu():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("GPU present")
    with pytest.raises(RuntimeError):
        ab.Context(0)


def test_cache_slot_count_matches_header():
    import re
    txt = open(ab.HEADER).read()
    assert int(re.search(r"#define ABCD_MAX_CACHE_SLOTS (\d+)", txt).group(1)) == ab.ABCD_MAX_CACHE_SLOTS


def test_cache_calls_reject_a_null_context(lib):
    # argument checks come before any CUDA call (no GPU needed)
    assert lib.abcd_cache_fetch(None, 0, None, None, 0) == ab.ABCD_ERR_INVALID_ARG
    assert lib.abcd_cache_wait(None, 0) == ab.ABCD_ERR_INVALID_ARG
    assert lib.abcd_cache_release(None, 0) == ab.ABCD_ERR_INVALID_ARG
    assert lib.abcd_cache_store(None, 0, None, None, 0) == ab.ABCD_ERR_INVALID_ARG
    assert lib.abcd_cache_sync(None) == ab.ABCD_ERR_INVALID_ARG
