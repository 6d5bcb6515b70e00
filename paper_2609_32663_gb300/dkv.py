"""Thin Python binding of the C ABI in include/dkv.h (libdkv.so).

Argument marshalling only: each function takes torch tensors (device buffers)
or numpy arrays (host inputs), passes raw pointers, sizes and the current CUDA
stream to the function of the same name in libdkv.so, and raises DkvError on a
non-zero status. Every step of the path runs in the library's CUDA kernels;
there is no Python or CPU fallback, and importing the functions fails loudly
when libdkv.so has not been built.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
# DKV_LIBRARY names another build of the same ABI to load instead, e.g. the
# bounds-checked libdkv_debug.so (build.build_library(debug=True)).
LIB_PATH = os.environ.get("DKV_LIBRARY") or os.path.join(_PKG, "libdkv.so")

DKV_OK, DKV_ERR_INVALID_ARG, DKV_ERR_CUDA, DKV_ERR_OOM, DKV_ERR_RANGE, DKV_ERR_TIMEOUT = range(6)
DKV_DEV_APPEND_OVERFLOW = 0x1
DKV_DEV_TMA_TIMEOUT = 0x2
DKV_DEV_MERGE_TIMEOUT = 0x4
DKV_DEV_BOUNDS = 0x8

# Every entry point include/dkv.h declares.
EXPORTS = ("dkv_last_error", "dkv_map_pattern", "dkv_plan_dense", "dkv_plan_query", "dkv_plan_read",
           "dkv_compact", "dkv_decode_attn", "dkv_decode_partial", "dkv_decode_combine", "dkv_advance",
           "dkv_plan_status", "dkv_free", "dkv_decode_attn_noalloc", "dkv_budget", "dkv_topk_workspace_bytes",
           "dkv_topk_mask", "dkv_decode_multi", "dkv_map_pattern_inplace", "dkv_compact_inplace",
           "dkv_vmm_alloc", "dkv_vmm_trim", "dkv_vmm_pages_to_keep", "dkv_vmm_mapped_bytes", "dkv_vmm_page_bytes",
           "dkv_vmm_free")


class DkvError(RuntimeError):
    def __init__(self, status, func, msg):
        super().__init__(f"{func} failed with status {status}: {msg}")
        self.status = status


class dkv_shape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("L", "H", "H_kv", "D", "head_dim", "sink", "recent", "bin_width")]


@dataclass(frozen=True)
class Shape:
    """Model and pattern geometry (dkv_shape)."""
    L: int
    H: int
    H_kv: int
    D: int
    head_dim: int = 128
    sink: int = 128
    recent: int = 1024
    bin_width: int = 128

    def c(self):
        return dkv_shape(self.L, self.H, self.H_kv, self.D, self.head_dim, self.sink, self.recent,
                         self.bin_width)

    @property
    def G(self):
        return self.H // self.H_kv


_lib = None


def lib(path: str | None = None):
    """Load libdkv.so (once) and declare its signatures."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is missing: build it with paper_2609_32663_gb300.build.build_library() "
                           "(or __graft_entry__.build()); there is no fallback path")
    L = ctypes.CDLL(p)
    V, I32, I64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    PP = ctypes.POINTER(ctypes.c_void_p)
    L.dkv_last_error.restype = ctypes.c_char_p
    L.dkv_last_error.argtypes = []
    L.dkv_map_pattern.restype = ctypes.c_int
    L.dkv_map_pattern.argtypes = [V, V, I32, ctypes.POINTER(dkv_shape), I32, V, PP]
    L.dkv_map_pattern_inplace.restype = ctypes.c_int
    L.dkv_map_pattern_inplace.argtypes = [V, V, I32, ctypes.POINTER(dkv_shape), I32, I64, V, PP]
    L.dkv_compact_inplace.restype = ctypes.c_int
    L.dkv_compact_inplace.argtypes = [V, V, V, V]
    L.dkv_vmm_alloc.restype = ctypes.c_int
    L.dkv_vmm_alloc.argtypes = [I64, PP, PP]
    L.dkv_vmm_trim.restype = ctypes.c_int
    L.dkv_vmm_trim.argtypes = [V, V, I32, ctypes.POINTER(I64)]
    L.dkv_vmm_pages_to_keep.restype = None
    L.dkv_vmm_pages_to_keep.argtypes = [V, I64, I64, I32, I32, I64, I64, I64, V]
    L.dkv_vmm_mapped_bytes.restype = I64
    L.dkv_vmm_mapped_bytes.argtypes = [V]
    L.dkv_vmm_page_bytes.restype = I64
    L.dkv_vmm_page_bytes.argtypes = [V]
    L.dkv_vmm_free.restype = None
    L.dkv_vmm_free.argtypes = [V]
    L.dkv_plan_dense.restype = ctypes.c_int
    L.dkv_plan_dense.argtypes = [V, I32, ctypes.POINTER(dkv_shape), I64, V, PP]
    L.dkv_plan_query.restype = ctypes.c_int
    L.dkv_plan_query.argtypes = [V, ctypes.POINTER(I64), ctypes.POINTER(I64), PP, PP, PP, PP]
    L.dkv_plan_read.restype = ctypes.c_int
    L.dkv_plan_read.argtypes = [V, V, V, V, V, V]
    L.dkv_compact.restype = ctypes.c_int
    L.dkv_compact.argtypes = [V, V, V, I64, V, V, V]
    L.dkv_decode_attn.restype = ctypes.c_int
    L.dkv_decode_attn.argtypes = [V, I32, V, V, V, V, V, V, ctypes.c_float, V, V]
    L.dkv_decode_multi.restype = ctypes.c_int
    L.dkv_decode_multi.argtypes = [V, I32, V, I32, V, V, V, ctypes.c_float, V, V]
    L.dkv_decode_partial.restype = ctypes.c_int
    L.dkv_decode_partial.argtypes = [V, I32, V, V, V, V, V, V, ctypes.c_float, V]
    L.dkv_decode_combine.restype = ctypes.c_int
    L.dkv_decode_combine.argtypes = [V, I32, V, I32, V, V]
    L.dkv_advance.restype = ctypes.c_int
    L.dkv_advance.argtypes = [V, V, V]
    L.dkv_plan_status.restype = ctypes.c_int
    L.dkv_plan_status.argtypes = [V, ctypes.POINTER(I32), I32, V]
    L.dkv_decode_attn_noalloc.restype = ctypes.c_int
    L.dkv_decode_attn_noalloc.argtypes = [ctypes.POINTER(dkv_shape), I32, I32, I32, V, V, V, V, V, V, V, V, V,
                                          ctypes.c_float, V, V, V]
    L.dkv_free.restype = None
    L.dkv_free.argtypes = [V]
    L.dkv_budget.restype = I64
    L.dkv_budget.argtypes = [ctypes.c_double, I32, I32, I32]
    L.dkv_topk_workspace_bytes.restype = I64
    L.dkv_topk_workspace_bytes.argtypes = []
    L.dkv_topk_mask.restype = ctypes.c_int
    L.dkv_topk_mask.argtypes = [V, I64, I64, V, V, I64, V]
    if path is None:
        _lib = L
    return L


def _check(status, func):
    if status != DKV_OK:
        raise DkvError(status, func, lib().dkv_last_error().decode(errors="replace"))


def _ptr(t):
    """Device (torch) or host (numpy) buffer -> address; None -> NULL."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _dev(t, name, dtypes=None, numel=None, min_numel=None):
    """Address of a device buffer argument, checked: a contiguous CUDA tensor of
    the expected element type and size (an int is taken as a raw device address,
    None as NULL). A host tensor passed here would make the kernel read host
    addresses, so it is refused before the call."""
    if t is None or isinstance(t, int):
        return t
    why = None
    if not getattr(t, "is_cuda", False):
        why = "must be a CUDA tensor"
    elif not t.is_contiguous():
        why = "must be contiguous"
    elif dtypes is not None and t.dtype not in dtypes:
        why = f"has dtype {t.dtype}, expected one of {dtypes}"
    elif numel is not None and t.numel() != numel:
        why = f"has {t.numel()} elements, expected {numel}"
    elif min_numel is not None and t.numel() < min_numel:
        why = f"has {t.numel()} elements, needs at least {min_numel}"
    if why:
        raise DkvError(DKV_ERR_INVALID_ARG, "argument check", f"{name} {why}")
    return t.data_ptr()


def _bf16():
    import torch
    return (torch.bfloat16, torch.int16)


def _i32():
    import torch
    return (torch.int32,)


def _f32():
    import torch
    return (torch.float32,)


def _stream(stream):
    if stream is None:
        import torch
        if not torch.cuda.is_available():
            return None
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


class Plan:
    """Owner of a dkv_plan*; dkv_free runs on close() or garbage collection."""

    def __init__(self, handle, shape: Shape, B: int, dense: bool):
        self.handle = handle
        self.shape = shape
        self.B = B
        self.dense = dense

    def close(self):
        if self.handle:
            lib().dkv_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def _as_parameter_(self):
        if not self.handle:
            raise ValueError("plan already freed")
        return ctypes.c_void_p(self.handle)


def dkv_map_pattern(M, ctx_len, shape: Shape, reserve_rows: int = 0, stream=None) -> Plan:
    M = np.ascontiguousarray(M, dtype=np.uint8)
    ctx = np.ascontiguousarray(ctx_len, dtype=np.int32)
    out = ctypes.c_void_p()
    sh = shape.c()
    _check(lib().dkv_map_pattern(_ptr(M), _ptr(ctx), len(ctx), ctypes.byref(sh), int(reserve_rows),
                                 _stream(stream), ctypes.byref(out)), "dkv_map_pattern")
    return Plan(out.value, shape, len(ctx), False)


def dkv_map_pattern_inplace(M, ctx_len, shape: Shape, T_stride: int, reserve_rows: int = 0, stream=None) -> Plan:
    """dkv_map_pattern with every slab at the start of its own dense region (off[h] = h T_stride)."""
    M = np.ascontiguousarray(M, dtype=np.uint8)
    ctx = np.ascontiguousarray(ctx_len, dtype=np.int32)
    out = ctypes.c_void_p()
    sh = shape.c()
    _check(lib().dkv_map_pattern_inplace(_ptr(M), _ptr(ctx), len(ctx), ctypes.byref(sh), int(reserve_rows),
                                         int(T_stride), _stream(stream), ctypes.byref(out)), "dkv_map_pattern_inplace")
    return Plan(out.value, shape, len(ctx), False)


def dkv_compact_inplace(plan: Plan, K, V, stream=None):
    """Move each slab's kept rows to the start of its region of K and V (in place)."""
    need = dkv_plan_query(plan).total_rows * 128
    _check(lib().dkv_compact_inplace(plan, _dev(K, "K", _bf16(), min_numel=need), _dev(V, "V", _bf16(), min_numel=need),
                                     _stream(stream)), "dkv_compact_inplace")


class VmmBuffer:
    """A page-backed device buffer (dkv_vmm_alloc); .tensor(shape, dtype) views it as a torch tensor."""

    def __init__(self, nbytes: int):
        h, p = ctypes.c_void_p(), ctypes.c_void_p()
        _check(lib().dkv_vmm_alloc(int(nbytes), ctypes.byref(h), ctypes.byref(p)), "dkv_vmm_alloc")
        self.handle, self.ptr, self.nbytes = h.value, p.value, int(nbytes)

    @property
    def _as_parameter_(self):
        return ctypes.c_void_p(self.handle)

    def tensor(self, shape, dtype):
        import torch
        typestr = {torch.bfloat16: "<i2", torch.int16: "<i2", torch.float32: "<f4", torch.uint8: "|u1"}[dtype]
        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        assert n <= self.nbytes

        class _View:
            __cuda_array_interface__ = {"shape": tuple(int(x) for x in shape), "typestr": typestr,
                                        "data": (self.ptr, False), "version": 3}
        t = torch.as_tensor(_View(), device="cuda")
        return t.view(torch.bfloat16) if dtype == torch.bfloat16 else t

    def trim(self, plan, guard_rows: int = 16) -> int:
        freed = ctypes.c_int64()
        _check(lib().dkv_vmm_trim(self, plan, int(guard_rows), ctypes.byref(freed)), "dkv_vmm_trim")
        return freed.value

    def mapped_bytes(self) -> int:
        return int(lib().dkv_vmm_mapped_bytes(self))

    def page_bytes(self) -> int:
        return int(lib().dkv_vmm_page_bytes(self))

    def close(self):
        if self.handle:
            lib().dkv_vmm_free(self)
            self.handle = None


def dkv_vmm_pages_to_keep(len_host, T_stride: int, reserve: int, guard_rows: int, page_bytes: int, npages: int,
                          row_bytes: int = 256) -> np.ndarray:
    ln = np.ascontiguousarray(len_host, np.int32)
    keep = np.zeros(max(npages, 1), np.uint8)
    lib().dkv_vmm_pages_to_keep(_ptr(ln), ln.size, int(T_stride), int(reserve), int(guard_rows), int(row_bytes),
                                int(page_bytes), int(npages), _ptr(keep))
    return keep[:npages]


def dkv_plan_dense(ctx_len, shape: Shape, T_stride: int, stream=None) -> Plan:
    ctx = np.ascontiguousarray(ctx_len, dtype=np.int32)
    out = ctypes.c_void_p()
    sh = shape.c()
    _check(lib().dkv_plan_dense(_ptr(ctx), len(ctx), ctypes.byref(sh), int(T_stride), _stream(stream),
                                ctypes.byref(out)), "dkv_plan_dense")
    return Plan(out.value, shape, len(ctx), True)


@dataclass
class PlanInfo:
    total_rows: int
    kept_rows: int
    d_len: int
    d_off: int
    d_ioff: int | None
    d_idx: int | None


def dkv_plan_query(plan: Plan) -> PlanInfo:
    tr, kr = ctypes.c_int64(), ctypes.c_int64()
    pl, po, pi, px = (ctypes.c_void_p() for _ in range(4))
    _check(lib().dkv_plan_query(plan, ctypes.byref(tr), ctypes.byref(kr), ctypes.byref(pl),
                                ctypes.byref(po), ctypes.byref(pi), ctypes.byref(px)), "dkv_plan_query")
    return PlanInfo(tr.value, kr.value, pl.value, po.value, pi.value, px.value)


def dkv_compact(plan: Plan, K, V, Kc, Vc, T_stride: int | None = None, stream=None):
    if T_stride is None:
        T_stride = K.shape[-2]
    sh = plan.shape
    dense = sh.L * plan.B * sh.H_kv * int(T_stride) * 128
    packed = dkv_plan_query(plan).total_rows * 128
    _check(lib().dkv_compact(plan, _dev(K, "K", _bf16(), min_numel=dense), _dev(V, "V", _bf16(), min_numel=dense),
                             int(T_stride), _dev(Kc, "Kc", _bf16(), min_numel=packed),
                             _dev(Vc, "Vc", _bf16(), min_numel=packed), _stream(stream)), "dkv_compact")


def _decode_ptrs(plan: Plan, q, k_new, v_new, n_appended, Kc, Vc, Q: int = 1):
    sh, B = plan.shape, plan.B
    rows = dkv_plan_query(plan).total_rows * 128
    return (_dev(q, "q", _bf16(), numel=B * Q * sh.H * 128),
            _dev(k_new, "k_new", _bf16(), numel=B * sh.H_kv * 128),
            _dev(v_new, "v_new", _bf16(), numel=B * sh.H_kv * 128),
            _dev(n_appended, "n_appended", _i32(), numel=B),
            _dev(Kc, "Kc", _bf16(), min_numel=rows), _dev(Vc, "Vc", _bf16(), min_numel=rows))


def dkv_decode_attn(plan: Plan, layer: int, q, k_new, v_new, n_appended, Kc, Vc, out, scale: float = 0.0,
                    stream=None):
    qp, kp, vp, np_, kc, vc = _decode_ptrs(plan, q, k_new, v_new, n_appended, Kc, Vc)
    op = _dev(out, "out", _f32(), numel=plan.B * plan.shape.H * 128)
    _check(lib().dkv_decode_attn(plan, int(layer), qp, kp, vp, np_, kc, vc, ctypes.c_float(scale), op,
                                 _stream(stream)), "dkv_decode_attn")


def dkv_decode_multi(plan: Plan, layer: int, q, num_queries: int, n_appended, Kc, Vc, out, scale: float = 0.0,
                     stream=None):
    """num_queries queries per sequence over the same compressed rows: q bf16
    [B][Q][H][128] -> out fp32 [B][Q][H][128]."""
    Q = max(int(num_queries), 1)
    qp, _, _, np_, kc, vc = _decode_ptrs(plan, q, None, None, n_appended, Kc, Vc, Q=Q)
    op = _dev(out, "out", _f32(), numel=plan.B * Q * plan.shape.H * 128)
    _check(lib().dkv_decode_multi(plan, int(layer), qp, int(num_queries), np_, kc, vc, ctypes.c_float(scale), op,
                                  _stream(stream)), "dkv_decode_multi")


def dkv_decode_partial(plan: Plan, layer: int, q, k_new, v_new, n_appended, Kc, Vc, scale: float = 0.0,
                       stream=None):
    qp, kp, vp, np_, kc, vc = _decode_ptrs(plan, q, k_new, v_new, n_appended, Kc, Vc)
    _check(lib().dkv_decode_partial(plan, int(layer), qp, kp, vp, np_, kc, vc, ctypes.c_float(scale),
                                    _stream(stream)), "dkv_decode_partial")


def dkv_decode_combine(plan: Plan, layer: int, n_appended, with_new_token: bool, out, stream=None):
    np_ = _dev(n_appended, "n_appended", _i32(), numel=plan.B)
    op = _dev(out, "out", _f32(), numel=plan.B * plan.shape.H * 128)
    _check(lib().dkv_decode_combine(plan, int(layer), np_, int(bool(with_new_token)), op, _stream(stream)),
           "dkv_decode_combine")


def dkv_advance(plan: Plan, n_appended, stream=None):
    _check(lib().dkv_advance(plan, _dev(n_appended, "n_appended", _i32(), numel=plan.B), _stream(stream)),
           "dkv_advance")


def dkv_plan_status(plan: Plan, clear: bool = False, stream=None) -> int:
    w = ctypes.c_int32()
    _check(lib().dkv_plan_status(plan, ctypes.byref(w), int(bool(clear)), _stream(stream)), "dkv_plan_status")
    return w.value


def dkv_free(plan: Plan):
    plan.close()


def dkv_budget(rho: float, L: int, H: int, D: int) -> int:
    """K_rho = round(rho L H D) (App. A.3); raises on bad arguments."""
    k = lib().dkv_budget(float(rho), int(L), int(H), int(D))
    if k < 0:
        raise DkvError(1, "dkv_budget", f"rho={rho} L={L} H={H} D={D}")
    return int(k)


def dkv_topk_workspace_bytes() -> int:
    return int(lib().dkv_topk_workspace_bytes())


def dkv_topk_mask(P, K: int, M, workspace, stream=None):
    """M (device uint8, same element count as P) = TopKMask(P, K) of Eq. 3."""
    import torch
    n = P.numel()
    pp = _dev(P, "P", _f32())
    mp = _dev(M, "M", (torch.uint8,), numel=n)
    wp = _dev(workspace, "workspace")
    nbytes = workspace.numel() * workspace.element_size()
    _check(lib().dkv_topk_mask(pp, int(n), int(K), mp, wp, int(nbytes), _stream(stream)), "dkv_topk_mask")


def dkv_decode_attn_noalloc(shape: Shape, B: int, layer: int, reserve_rows: int, d_len, d_off, d_ioff, q, k_new,
                            v_new, n_appended, Kc, Vc, out, scale: float = 0.0, status=None, stream=None):
    """Decode attention that allocates no device memory; d_len/d_off/d_ioff are
    device addresses (ints) or tensors of the plan metadata."""
    sh = shape.c()
    _check(lib().dkv_decode_attn_noalloc(
        ctypes.byref(sh), int(B), int(layer), int(reserve_rows), _dev(d_len, "d_len"), _dev(d_off, "d_off"),
        _dev(d_ioff, "d_ioff"), _dev(q, "q", _bf16(), numel=B * shape.H * 128),
        _dev(k_new, "k_new", _bf16(), numel=B * shape.H_kv * 128), _dev(v_new, "v_new", _bf16(), numel=B * shape.H_kv * 128),
        _dev(n_appended, "n_appended", _i32(), numel=B), _dev(Kc, "Kc", _bf16()), _dev(Vc, "Vc", _bf16()),
        ctypes.c_float(scale), _dev(out, "out", _f32(), numel=B * shape.H * 128), _dev(status, "status", _i32()),
        _stream(stream)), "dkv_decode_attn_noalloc")


def dkv_plan_read(plan: Plan, stream=None):
    """Host copies (numpy) of the plan's len, off, ioff and idx arrays."""
    info = dkv_plan_query(plan)
    NH = plan.shape.L * plan.B * plan.shape.H_kv
    ln = np.zeros(NH, np.int32)
    off = np.zeros(NH + 1, np.int64)
    ioff = np.zeros(NH + 1, np.int64)
    idx = np.zeros(max(info.kept_rows, 1), np.int32)
    _check(lib().dkv_plan_read(plan, _ptr(ln), _ptr(off), _ptr(ioff), _ptr(idx), _stream(stream)),
           "dkv_plan_read")
    if plan.dense:
        return ln, off, None, None
    return ln, off, ioff, idx[: info.kept_rows]
