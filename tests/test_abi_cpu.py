"""The C ABI library builds, loads and exports every declared entry point, and its
host-side argument checks answer without a GPU (no kernel is launched here)."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def dkvmod():
    from paper_2609_32663_gb300 import build
    build.build_library()
    import paper_2609_32663_gb300.dkv as dkv
    return dkv


def declared_functions():
    src = open(os.path.join(ROOT, "include", "dkv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dkv_\w+)\s*\(", src)))


def test_header_declares_the_binding_exports(dkvmod):
    assert declared_functions() == sorted(dkvmod.EXPORTS)


def test_library_exports_every_declared_symbol(dkvmod):
    lib = ctypes.CDLL(dkvmod.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_library_is_built_for_sm_103a_only():
    from paper_2609_32663_gb300 import build
    assert build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]


def _shape(dkv, **kw):
    base = dict(L=2, H=8, H_kv=2, D=4, sink=2, recent=3, bin_width=5)
    base.update(kw)
    return dkv.Shape(**base)


@pytest.mark.parametrize("kw,ctx,status", [
    (dict(H=6, H_kv=4), [10], "INVALID_ARG"),           # H % H_kv != 0
    (dict(head_dim=64), [10], "INVALID_ARG"),            # only 128
    (dict(H=18, H_kv=2), [10], "INVALID_ARG"),           # group size 9 > 8
    (dict(bin_width=0), [10], "INVALID_ARG"),
    (dict(), [-1], "INVALID_ARG"),                       # negative length
    (dict(), [2 + 3 + 4 * 5 + 1], "RANGE"),              # needs a 5th bin
])
def test_map_pattern_rejects_bad_arguments(dkvmod, kw, ctx, status):
    dkv = dkvmod
    sh = _shape(dkv, **kw)
    M = np.zeros((sh.L, sh.H, sh.D), np.uint8)
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_map_pattern(M, ctx, sh, stream=0)
    assert e.value.status == getattr(dkv, "DKV_ERR_" + status)
    assert dkv.lib().dkv_last_error()


def test_map_pattern_rejects_non_binary_pattern(dkvmod):
    dkv = dkvmod
    sh = _shape(dkv)
    M = np.zeros((sh.L, sh.H, sh.D), np.uint8)
    M[1, 3, 2] = 7
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_map_pattern(M, [10], sh, stream=0)
    assert e.value.status == dkv.DKV_ERR_INVALID_ARG
    assert b"M[" in dkv.lib().dkv_last_error()


def test_null_arguments(dkvmod):
    dkv = dkvmod
    L = dkv.lib()
    out = ctypes.c_void_p(123)
    sh = _shape(dkv).c()
    assert L.dkv_map_pattern(None, None, 1, ctypes.byref(sh), 0, None, ctypes.byref(out)) == dkv.DKV_ERR_INVALID_ARG
    assert out.value is None
    assert L.dkv_map_pattern(None, None, 1, ctypes.byref(sh), 0, None, None) == dkv.DKV_ERR_INVALID_ARG
    assert L.dkv_compact(None, None, None, 1, None, None, None) == dkv.DKV_ERR_INVALID_ARG
    assert L.dkv_decode_attn(None, 0, None, None, None, None, None, None, ctypes.c_float(0), None, None) == \
        dkv.DKV_ERR_INVALID_ARG
    assert L.dkv_advance(None, None, None) == dkv.DKV_ERR_INVALID_ARG
    assert L.dkv_plan_query(None, None, None, None, None, None, None) == dkv.DKV_ERR_INVALID_ARG
    L.dkv_free(None)  # NULL-safe


def test_injected_allocation_failure_reports_oom(dkvmod, monkeypatch):
    """Host-side fault injection: the first device allocation fails before any
    CUDA call, and the error surfaces as DKV_ERR_OOM with a message."""
    dkv = dkvmod
    monkeypatch.setenv("DKV_FAULT", "alloc")
    sh = _shape(dkv)
    M = np.ones((sh.L, sh.H, sh.D), np.uint8)
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_map_pattern(M, [12, 20], sh, stream=0)
    assert e.value.status == dkv.DKV_ERR_OOM
    assert b"injected" in dkv.lib().dkv_last_error()


def test_dense_plan_rejects_short_stride(dkvmod):
    dkv = dkvmod
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_plan_dense([100, 300], _shape(dkv), T_stride=200, stream=0)
    assert e.value.status == dkv.DKV_ERR_INVALID_ARG


def test_binding_fails_loudly_without_library(tmp_path):
    import paper_2609_32663_gb300.dkv as dkv
    with pytest.raises(RuntimeError, match="missing"):
        dkv.lib(str(tmp_path / "libdkv.so"))


def test_budget_matches_oracle(dkvmod):
    """dkv_budget (host arithmetic of the library) against the oracle's budget."""
    import oracle as O
    rng = np.random.default_rng(3)
    cases = [(0.35, 32, 32, 1013), (0.5, 1, 1, 5), (0.5, 1, 1, 3), (0.0, 32, 32, 128), (1.0, 28, 28, 64)]
    cases += [(float(r), int(L), int(H), int(D)) for r, L, H, D in
              zip(rng.random(50), rng.integers(1, 80, 50), rng.integers(1, 64, 50), rng.integers(1, 2048, 50))]
    for rho, L, H, D in cases:
        assert dkvmod.dkv_budget(rho, L, H, D) == O.budget(rho, L, H, D), (rho, L, H, D)
    for bad in [(-0.01, 1, 1, 1), (1.01, 1, 1, 1), (float("nan"), 1, 1, 1), (0.5, -1, 1, 1)]:
        with pytest.raises(dkvmod.DkvError):
            dkvmod.dkv_budget(*bad)


def test_topk_rejects_bad_arguments(dkvmod):
    """Argument checks run before any launch (fake device addresses are never touched)."""
    L = dkvmod.lib()
    ws_need = L.dkv_topk_workspace_bytes()
    assert 0 < ws_need <= 64 * 1024
    fake = ctypes.c_void_p(0x1000)
    for n, K, P, M, ws, wsb in [(-1, 0, fake, fake, fake, ws_need), (1 << 31, 1, fake, fake, fake, ws_need),
                                (10, 11, fake, fake, fake, ws_need), (10, -1, fake, fake, fake, ws_need),
                                (10, 3, None, fake, fake, ws_need), (10, 3, fake, None, fake, ws_need),
                                (10, 3, fake, fake, None, ws_need), (10, 3, fake, fake, fake, ws_need - 4),
                                (10, 3, fake, fake, ctypes.c_void_p(0x1002), ws_need)]:
        assert L.dkv_topk_mask(P, n, K, M, ws, wsb, None) == 1, (n, K)
        assert L.dkv_last_error()


@pytest.mark.parametrize("page", [2 << 20, 65536, 1000])
def test_vmm_page_rule_keeps_every_needed_row(dkvmod, page):
    """dkv_vmm_pages_to_keep against an independent interval check: every byte a
    slab may still touch (len + reserve + guard rows, capped at its region) is in
    a kept page, and no page outside all of those is kept."""
    rng = np.random.default_rng(page)
    for trial in range(20):
        NH = int(rng.integers(1, 40))
        T = int(rng.integers(1, 20000))
        reserve, guard = int(rng.integers(0, 300)), int(rng.integers(16, 64))
        ln = rng.integers(0, T + 1, NH).astype(np.int32)
        ln[rng.random(NH) < 0.2] = 0
        total = NH * T * 256
        npages = -(-total // page)
        keep = dkvmod.dkv_vmm_pages_to_keep(ln, T, reserve, guard, page, npages)
        want = np.zeros(npages, np.uint8)
        for h in range(NH):
            rows = min(T, int(ln[h]) + reserve + guard)
            b0, b1 = h * T * 256, h * T * 256 + rows * 256
            if rows > 0:
                want[b0 // page:(b1 - 1) // page + 1] = 1
        assert np.array_equal(keep, want), trial
        for h in range(NH):  # the safety property itself
            rows = min(T, int(ln[h]) + reserve + guard)
            for b in (h * T * 256, h * T * 256 + rows * 256 - 1):
                if rows > 0:
                    assert keep[b // page] == 1


def test_binding_refuses_host_and_misshapen_buffers(dkvmod):
    """The binding passes device addresses only: a host tensor, a strided view,
    a wrong element type or a wrong size is refused with DKV_ERR_INVALID_ARG
    before the library is called (a host address would be read by a kernel)."""
    import torch
    dkv = dkvmod
    cases = [
        (torch.zeros(8, dtype=torch.float32), {}, "CUDA tensor"),
    ]
    for t, kw, msg in cases:
        with pytest.raises(dkv.DkvError) as e:
            dkv._dev(t, "out", **kw)
        assert e.value.status == dkv.DKV_ERR_INVALID_ARG and msg in str(e.value)

    class FakeCuda:
        """Stands in for a device tensor: the checks read only these fields."""
        is_cuda = True

        def __init__(self, dtype, n, contiguous=True):
            self.dtype, self.n, self.c = dtype, n, contiguous

        def is_contiguous(self):
            return self.c

        def numel(self):
            return self.n

        def data_ptr(self):
            return 0x7F0000000000

    f32 = (torch.float32,)
    for t, kw, msg in [
        (FakeCuda(torch.float32, 8, contiguous=False), {"dtypes": f32}, "contiguous"),
        (FakeCuda(torch.float16, 8), {"dtypes": f32}, "dtype"),
        (FakeCuda(torch.float32, 7), {"dtypes": f32, "numel": 8}, "expected 8"),
        (FakeCuda(torch.float32, 7), {"dtypes": f32, "min_numel": 8}, "at least 8"),
    ]:
        with pytest.raises(dkv.DkvError) as e:
            dkv._dev(t, "out", **kw)
        assert e.value.status == dkv.DKV_ERR_INVALID_ARG and msg in str(e.value)
    assert dkv._dev(FakeCuda(torch.float32, 8), "out", dtypes=f32, numel=8) == 0x7F0000000000
    assert dkv._dev(None, "k_new") is None
    assert dkv._dev(0x1000, "raw") == 0x1000


def test_header_is_plain_c_and_links_from_c(dkvmod, tmp_path):
    """include/dkv.h compiles as C11 (the CUDA runtime header it includes needs
    C11), and a C program that takes the address of every declared entry point
    links against libdkv.so and runs (no GPU call)."""
    import shutil
    import subprocess
    cc = os.environ.get("CC", "gcc")
    if shutil.which(cc) is None:
        pytest.skip("no C compiler")
    cuda_inc = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")
    names = declared_functions()
    prog = tmp_path / "abi.c"
    prog.write_text(
        '#include <stdio.h>\n#include "dkv.h"\n'
        "typedef void (*fn)(void);\nint main(void) {\n    const fn f[] = {\n"
        + "".join(f"        (fn)&{n},\n" for n in names)
        + "    };\n    int n = 0;\n"
        "    for (unsigned i = 0; i < sizeof f / sizeof f[0]; ++i) n += f[i] != 0;\n"
        '    printf("%d\\n", n);\n    return 0;\n}\n')
    libdir = os.path.dirname(dkvmod.LIB_PATH)
    exe = tmp_path / "abi"
    subprocess.check_call([cc, "-std=c11", "-Wall", "-Wextra", "-Werror",
                           "-I", os.path.join(ROOT, "include"), "-I", cuda_inc, str(prog), "-o", str(exe),
                           "-L", libdir, "-ldkv", f"-Wl,-rpath,{libdir}"])
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    assert int(out) == len(names)


def test_bounds_checked_build_exports_every_declared_symbol(dkvmod):
    """The -DDKV_DEBUG variant (libdkv_debug.so) compiles from the same sources
    and exports the same ABI; its kernels run in tests/test_gpu_bounds_build.py."""
    from paper_2609_32663_gb300 import build
    lib = ctypes.CDLL(build.build_library(debug=True))
    for name in declared_functions():
        assert hasattr(lib, name), name
