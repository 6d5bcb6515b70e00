"""The oracle and the product path stay independent: neither imports, includes
or links the other, and the only module both read is the seeded input generator
(which holds none of the method's arithmetic). CPU only: reads the sources."""
import ast
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2609_32663_gb300")
ORACLE = os.path.join(ROOT, "oracle")


def _py_imports(path):
    tree = ast.parse(open(path).read(), filename=path)
    names = set()
    for node in ast.walk(tree):
        if isinstance(node, ast.Import):
            names.update(a.name.split(".")[0] for a in node.names)
        elif isinstance(node, ast.ImportFrom) and node.module and node.level == 0:
            names.add(node.module.split(".")[0])
    return names


def _files(d, exts):
    return sorted(os.path.join(d, f) for f in os.listdir(d) if f.endswith(exts))


def test_product_python_never_imports_the_oracle():
    for f in _files(PKG, (".py",)):
        assert "oracle" not in _py_imports(f), f


def test_product_sources_include_only_their_own_headers():
    srcs = _files(os.path.join(PKG, "csrc"), (".cu", ".cuh"))
    assert srcs
    own = {os.path.basename(f) for f in srcs} | {"dkv.h"}
    for f in srcs:
        for inc in re.findall(r'#include\s+"([^"]+)"', open(f).read()):
            assert os.path.basename(inc) in own, (f, inc)
            assert "oracle" not in inc, (f, inc)


def test_product_build_does_not_compile_or_link_the_oracle():
    src = open(os.path.join(PKG, "build.py")).read()
    assert "oracle" not in src


def test_oracle_imports_nothing_from_the_product():
    for f in _files(ORACLE, (".py",)):
        assert "paper_2609_32663_gb300" not in _py_imports(f), f
    c = open(os.path.join(ORACLE, "dkv_oracle.c")).read()
    assert re.findall(r'#include\s+"([^"]+)"', c) == []
    for inc in re.findall(r"#include\s+<([^>]+)>", c):
        assert inc in {"math.h", "stdint.h", "stdlib.h", "string.h"}, inc


def test_shared_input_module_holds_no_method_arithmetic():
    """inputs.py draws seeded tensors and patterns. The keep rule (distance bins
    and the retention mask), the union of positions over a group, the pack and
    the attention live only in the oracle and the kernels."""
    imports = _py_imports(os.path.join(PKG, "inputs.py"))
    assert "oracle" not in imports
    assert not imports & {"ctypes"}
    src = open(os.path.join(PKG, "inputs.py")).read()
    for word in ("softmax", "dkv_decode", "dkv_compact", "dkv_map_pattern", "bin_width", "keep_pos"):
        assert word not in src, word


# The generators reach exact budgets with three helpers that resemble steps of
# the method: a stable global top-k of scores (the shape of the pattern export),
# floor(x + 1/2) (the export's budget rounding) and a count of group columns
# with any head on (the size of the GQA union at full coverage). They only size
# and select generated patterns.
GENERATOR_ONLY = ("_gen_top_entries", "_gen_round", "_gen_group_columns")


def test_generator_only_helpers_are_private_to_the_generators():
    import paper_2609_32663_gb300.inputs as I
    for name in GENERATOR_ONLY:
        assert hasattr(I, name), name
        assert name not in I.__all__, name
    for name in ("topk_mask", "round_half_up", "_union_count"):
        assert not hasattr(I, name), name


def test_no_expected_value_comes_from_the_generator_helpers():
    """No test, smoke() or bench.py leg calls them: every expected mask, map,
    byte and output is the oracle's (or a hand-worked fixture's)."""
    users = _files(os.path.join(ROOT, "tests"), (".py",)) + [os.path.join(ROOT, "__graft_entry__.py"),
                                                            os.path.join(ROOT, "bench.py")]
    for f in users:
        if os.path.basename(f) == "test_separation_cpu.py":
            continue
        src = open(f).read()
        for name in GENERATOR_ONLY:
            assert name not in src, (f, name)
