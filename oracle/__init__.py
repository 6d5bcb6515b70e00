"""Python face of the Distance-KV CPU oracle (oracle/dkv_oracle.c).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import this module. The product library never
does, and this module imports nothing from the product package.

Every function is a thin ctypes call into the scalar fp64 C oracle, which states
Sec. 3.4 of the paper (Eq. 4 distance bin, Eq. 5 retention mask, the GQA union,
the ordered prune-and-pack, and decode attention over the packed cache).
bf16 tensors travel as uint16 bit patterns.
"""
import ctypes
from dataclasses import dataclass

import numpy as np

from . import build as _build

OK, ERR_INVALID_ARG, ERR_RANGE = 0, 1, 4

_lib = None


class _Shape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("L", "H", "Hkv", "D", "head_dim", "sink", "recent", "bin_width")]


@dataclass(frozen=True)
class Geometry:
    """L layers, H query heads, Hkv KV heads, D bins, sink S, recent R, bin width W."""
    L: int
    H: int
    Hkv: int
    D: int
    head_dim: int = 128
    sink: int = 128
    recent: int = 1024
    bin_width: int = 128

    def c(self):
        return _Shape(self.L, self.H, self.Hkv, self.D, self.head_dim, self.sink,
                      self.recent, self.bin_width)


def configure(L):
    """Declare the C signatures on a loaded oracle library."""
    P = ctypes.c_void_p
    L.oracle_distance_bin.restype = ctypes.c_long
    L.oracle_distance_bin.argtypes = [ctypes.c_long, ctypes.c_long, ctypes.POINTER(_Shape)]
    L.oracle_keep_logical.argtypes = [P, ctypes.POINTER(_Shape), ctypes.c_int, ctypes.c_int,
                                      ctypes.c_long, ctypes.c_long]
    L.oracle_keep_physical.argtypes = L.oracle_keep_logical.argtypes
    L.oracle_validate.argtypes = [P, P, ctypes.c_int, ctypes.POINTER(_Shape), ctypes.c_int]
    L.oracle_map.argtypes = [P, P, ctypes.c_int, ctypes.POINTER(_Shape), ctypes.c_int,
                             P, P, P, P]
    L.oracle_compact.argtypes = [P, P, P, P, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                 ctypes.c_int, ctypes.c_int64, P, P, P, P]
    L.oracle_attend.restype = None
    L.oracle_attend.argtypes = [P, P, P, ctypes.c_long, ctypes.c_int, ctypes.c_int,
                                ctypes.c_double, P, P]
    L.oracle_append.argtypes = [P, P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                ctypes.c_int, P, P, P, P, P]
    L.oracle_budget.restype = ctypes.c_long
    L.oracle_budget.argtypes = [ctypes.c_double, ctypes.c_long, ctypes.c_long, ctypes.c_long]
    L.oracle_topk_mask.argtypes = [P, ctypes.c_long, ctypes.c_long, P]
    L.oracle_decode.restype = None
    L.oracle_decode.argtypes = [P, P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                ctypes.c_int, P, P, P, P, ctypes.c_double, P]
    return L


def lib():
    global _lib
    if _lib is None:
        _lib = configure(ctypes.CDLL(_build.build()))
    return _lib


def use_library(path):
    """Point this module at another build of the oracle source (used by the
    mutation test to check that the pins reject planted mistakes). Returns the
    previously active library handle."""
    global _lib
    prev = _lib
    _lib = configure(ctypes.CDLL(path)) if isinstance(path, str) else path
    return prev


def _p(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class OracleError(RuntimeError):
    def __init__(self, code, what):
        super().__init__(f"{what}: oracle status {code}")
        self.code = code


def distance_bin(p, Tc, geo: Geometry):
    return lib().oracle_distance_bin(p, Tc, ctypes.byref(geo.c()))


def keep_logical(M, geo: Geometry, layer, h, p, Tc):
    M = _c(M, np.uint8)
    return lib().oracle_keep_logical(_p(M), ctypes.byref(geo.c()), layer, h, p, Tc)


def keep_physical(M, geo: Geometry, layer, g, p, Tc):
    M = _c(M, np.uint8)
    return lib().oracle_keep_physical(_p(M), ctypes.byref(geo.c()), layer, g, p, Tc)


def validate(M, Tc, geo: Geometry, reserve=0):
    M = _c(M, np.uint8)
    Tc = _c(Tc, np.int32)
    return lib().oracle_validate(_p(M), _p(Tc), len(Tc), ctypes.byref(geo.c()), reserve)


@dataclass
class Mapping:
    len: np.ndarray   # int32 [L*B*Hkv]
    off: np.ndarray   # int64 [NH+1], slab starts in the packed cache (slab = len + reserve rows)
    ioff: np.ndarray  # int64 [NH+1], slab starts in idx
    idx: np.ndarray   # int32 [sum len], kept positions, ascending per slab

    @property
    def total_rows(self):
        return int(self.off[-1])

    @property
    def kept_rows(self):
        return int(self.ioff[-1])


def map_pattern(M, Tc, geo: Geometry, reserve=0, with_idx=True) -> Mapping:
    """Eqs. 4-5 and the GQA union for every (layer, sequence, KV head)."""
    M = _c(M, np.uint8)
    Tc = _c(Tc, np.int32)
    B = len(Tc)
    NH = geo.L * B * geo.Hkv
    ln = np.zeros(NH, np.int32)
    off = np.zeros(NH + 1, np.int64)
    ioff = np.zeros(NH + 1, np.int64)
    shape = geo.c()
    rc = lib().oracle_map(_p(M), _p(Tc), B, ctypes.byref(shape), reserve,
                          _p(ln), _p(off), _p(ioff), None)
    if rc != OK:
        raise OracleError(rc, "oracle_map")
    idx = None
    if with_idx:
        idx = np.zeros(max(int(ioff[-1]), 1), np.int32)
        rc = lib().oracle_map(_p(M), _p(Tc), B, ctypes.byref(shape), reserve,
                              _p(ln), _p(off), _p(ioff), _p(idx))
        if rc != OK:
            raise OracleError(rc, "oracle_map")
        idx = idx[: int(ioff[-1])]
    return Mapping(ln, off, ioff, idx)


def compact(m: Mapping, geo_L, B, Hkv, K, V, T_stride, head_dim=128):
    """Ordered prune-and-pack of dense bf16 (uint16) K, V [L][B][Hkv][T_stride][hd]."""
    K = _c(K, np.uint16)
    V = _c(V, np.uint16)
    Kc = np.zeros((m.total_rows, head_dim), np.uint16)
    Vc = np.zeros((m.total_rows, head_dim), np.uint16)
    idx = m.idx if m.idx is not None and len(m.idx) else np.zeros(1, np.int32)
    rc = lib().oracle_compact(_p(m.len), _p(m.off), _p(m.ioff), _p(_c(idx, np.int32)),
                              geo_L, B, Hkv, head_dim, T_stride, _p(K), _p(V), _p(Kc), _p(Vc))
    if rc != OK:
        raise OracleError(rc, "oracle_compact")
    return Kc, Vc


def attend(q, Krows, Vrows, scale=None, with_weights=False):
    """fp64 softmax attention of G bf16 query rows over n bf16 K/V rows."""
    q = _c(q, np.uint16)
    G, hd = q.shape
    Krows = _c(Krows, np.uint16).reshape(-1, hd)
    Vrows = _c(Vrows, np.uint16).reshape(-1, hd)
    n = Krows.shape[0]
    scale = 1.0 / np.sqrt(hd) if scale is None or scale <= 0 else float(scale)
    out = np.zeros((G, hd), np.float64)
    w = np.zeros((G, max(n, 1)), np.float64) if with_weights else None
    lib().oracle_attend(_p(q), _p(Krows), _p(Vrows), n, G, hd, scale, _p(out), _p(w))
    if with_weights:
        return out, w[:, :n]
    return out


def append(m: Mapping, layer, B, Hkv, reserve, n_app, k_new, v_new, Kc, Vc, head_dim=128):
    """Write k_new/v_new [B][Hkv][hd] at row off+len+n_app[b] of each slab (in place)."""
    n_app = _c(n_app, np.int32)
    assert Kc.flags.c_contiguous and Vc.flags.c_contiguous and Kc.dtype == np.uint16
    rc = lib().oracle_append(_p(m.len), _p(m.off), layer, B, Hkv, head_dim, reserve, _p(n_app),
                             _p(_c(k_new, np.uint16)), _p(_c(v_new, np.uint16)), _p(Kc), _p(Vc))
    if rc != OK:
        raise OracleError(rc, "oracle_append")


def decode(m: Mapping, layer, B, H, Hkv, q, Kc, Vc, n_rows_app=None, scale=None, head_dim=128):
    """fp64 decode attention of layer `layer`: out [B][H][hd]."""
    q = _c(q, np.uint16)
    Kc = _c(Kc, np.uint16)
    Vc = _c(Vc, np.uint16)
    scale = 1.0 / np.sqrt(head_dim) if scale is None or scale <= 0 else float(scale)
    out = np.zeros((B, H, head_dim), np.float64)
    na = None if n_rows_app is None else _c(n_rows_app, np.int32)
    lib().oracle_decode(_p(m.len), _p(m.off), layer, B, H, Hkv, head_dim, _p(na), _p(q),
                        _p(Kc), _p(Vc), scale, _p(out))
    return out


def budget(rho, L, H, D):
    """K_rho = round(rho L H D) of App. A.3 (round = floor(x + 1/2)); -1 for bad arguments."""
    return lib().oracle_budget(float(rho), int(L), int(H), int(D))


def topk_mask(P, K):
    """Global Top-K mask of Eq. 3: uint8 array shaped like P with the K first entries
    (larger value first, ties to the lower flat index, NaN last) set to 1."""
    P = _c(P, np.float32)
    flat = P.reshape(-1)
    M = np.zeros(max(flat.size, 1), np.uint8)
    rc = lib().oracle_topk_mask(_p(flat), flat.size, int(K), _p(M))
    if rc != OK:
        raise OracleError(rc, "oracle_topk_mask")
    return M[: flat.size].reshape(P.shape)


__all__ = ["Geometry", "Mapping", "OracleError", "distance_bin", "keep_logical",
           "keep_physical", "validate", "map_pattern", "compact", "attend", "append", "decode",
           "budget", "topk_mask", "OK", "ERR_INVALID_ARG", "ERR_RANGE"]
