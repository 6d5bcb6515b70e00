"""Saved patterns: the file round-trips M bit for bit with its geometry, and a
pattern is refused when it is not 0/1 or is mapped with another geometry."""
import numpy as np
import pytest

from paper_2609_32663_gb300 import inputs as I
from paper_2609_32663_gb300.patterns import check_geometry, load_pattern, save_pattern


def test_round_trip(tmp_path):
    wl = I.WORKLOADS["llama8b-128k"]
    M = I.make_pattern(wl)
    p = tmp_path / "m.npz"
    save_pattern(p, M, wl.sink, wl.recent, wl.W, {"workload": wl.name, "seed": wl.seed})
    M2, geo, meta = load_pattern(p)
    assert M2.dtype == np.uint8 and np.array_equal(M2, M)
    assert geo == {"sink": wl.sink, "recent": wl.recent, "bin_width": wl.W}
    assert meta == {"workload": wl.name, "seed": wl.seed}


def test_rejects_non_binary_and_bad_shape(tmp_path):
    with pytest.raises(ValueError):
        save_pattern(tmp_path / "a.npz", np.full((2, 2, 2), 2, np.uint8), 128, 1024, 128)
    with pytest.raises(ValueError):
        save_pattern(tmp_path / "b.npz", np.zeros((2, 2), np.uint8), 128, 1024, 128)


def test_geometry_mismatch_is_refused(tmp_path):
    class Shape:
        L, H, D, sink, recent, bin_width = 1, 2, 3, 128, 1024, 64
    save_pattern(tmp_path / "c.npz", np.ones((1, 2, 3), np.uint8), 128, 1024, 128)
    _, geo, _ = load_pattern(tmp_path / "c.npz")
    with pytest.raises(ValueError):
        check_geometry(geo, Shape)
    Shape.bin_width = 128
    check_geometry(geo, Shape)
