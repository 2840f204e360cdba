"""The CUDA path and the oracle share no code, and the product path has no
fallback (CPU only).

Parity against the oracle proves something only if the two sides are
independent: neither may import, include or link the other, and the only
module both read is the seeded input generator.  The product path must fail
loudly when libeti is missing instead of computing anything on the host.
"""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _files(sub, exts):
    out = []
    for d, _, names in os.walk(os.path.join(ROOT, sub)):
        if "_build" in d or "__pycache__" in d:
            continue
        out += [os.path.join(d, n) for n in names if n.endswith(exts)]
    assert out, sub
    return out


def _code(path):
    txt = open(path).read()
    if path.endswith(".py"):
        txt = re.sub(r'"""[\s\S]*?"""', "", txt)
        return "\n".join(l.split("#")[0] for l in txt.splitlines())
    txt = re.sub(r"/\*[\s\S]*?\*/", "", txt)
    return "\n".join(l.split("//")[0] for l in txt.splitlines())


def test_product_path_never_reaches_the_oracle():
    for f in _files("paper_2603_03310_gb300", (".py", ".cu", ".cuh", ".h")) + _files("include", (".h",)):
        code = _code(f)
        assert not re.search(r"\bimport\s+oracle\b|\bfrom\s+oracle\b|eti_oracle", code), f


def test_oracle_never_reaches_the_cuda_path():
    for f in _files("oracle", (".py", ".c", ".h")):
        code = _code(f)
        assert not re.search(r"paper_2603_03310_gb300|libeti|eti\.h|csrc|\bcuda", code, re.I), f


def test_input_generators_hold_no_method_code():
    for f in _files("workloads", (".py",)):
        code = _code(f)
        assert not re.search(r"\boracle\b|paper_2603_03310_gb300", code), f
        # no entropy, softmax, attention or sampling arithmetic
        assert not re.search(r"softmax|entropy\(|log_softmax|scaled_dot_product|argmax", code), f


def test_bench_runs_the_oracle_only_in_its_cpu_legs():
    import ast
    tree = ast.parse(open(os.path.join(ROOT, "bench.py")).read())
    users = set()
    for fn in ast.walk(tree):
        if isinstance(fn, ast.FunctionDef):
            for node in ast.walk(fn):
                if isinstance(node, ast.Import) and any(a.name == "oracle" for a in node.names):
                    users.add(fn.name)
    assert users == {"oracle_step", "_oracle_sample", "cpu_baseline", "run_reference"}
    top = [n for n in tree.body if isinstance(n, (ast.Import, ast.ImportFrom))]
    assert not any(getattr(n, "module", None) == "oracle" or
                   any(a.name == "oracle" for a in n.names) for n in top)


def test_binding_refuses_to_run_without_the_library(tmp_path):
    import paper_2603_03310_gb300 as eti
    saved = eti._lib
    eti._lib = None
    try:
        with pytest.raises(eti.EtiError, match="not built"):
            eti.load(str(tmp_path / "libeti.so"))
    finally:
        eti._lib = saved
