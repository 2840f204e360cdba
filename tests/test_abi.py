"""The C-ABI library builds, loads and exports every symbol include/eti.h
declares; host-side argument validation rejects bad calls before anything is
enqueued.  CPU only: no call here reaches a kernel launch."""
import ctypes
import os
import re

import pytest

import paper_2603_03310_gb300 as eti
from paper_2603_03310_gb300 import buildlib as eti_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    eti_build.build()
    return eti.load()


def _declared():
    txt = open(os.path.join(ROOT, "include", "eti.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(eti_\w+)\s*\(", txt)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert {"eti_entropy_temp_sample", "eti_score_prune_blocks", "eti_paged_decode"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n
    assert set(eti.SYMBOLS) <= set(names)


def test_library_is_built_for_sm103a_only():
    import shutil, subprocess
    tool = shutil.which("cuobjdump") or "/usr/local/cuda/bin/cuobjdump"
    if not os.path.exists(tool):
        pytest.skip("cuobjdump not available")
    # list the embedded ELF architectures (names only; nothing is disassembled)
    p = subprocess.run([tool, "--list-elf", eti.LIB_PATH], capture_output=True, text=True)
    archs = set(re.findall(r"sm_\w+", p.stdout))
    assert archs == {"sm_103a"}, archs


def test_version_and_status_strings(lib):
    assert "libeti" in eti.version()
    for s in (0, -1, -2, -3, -4, -5, -6):
        assert lib.eti_status_string(s).decode()


def test_ctrl_defaults(lib):
    p = eti.ctrl_params()
    assert (p.eta, p.sign, p.T_min, p.T_max, p.eps_H, p.H_min, p.theta_hi) == \
        pytest.approx((0.1, -1.0, 0.05, 5.0, 0.0, 0.0, 1.0))
    assert p.theta_user == float("inf")
    assert (p.T_cal, p.rho_T, p.dtheta) == (1.0, 0.0, 0.0)     # guards off by default


NULL = None


def test_entropy_call_validation(lib):
    P = ctypes.c_void_p
    fake = P(256)
    prm = eti.ctrl_params()
    f = lib.eti_entropy_temp_sample
    ws = lib.eti_entropy_temp_sample_workspace_size(4, 10)
    assert ws > 0
    # tok, H, T_out, dH, theta_next, tok_surprisal, surp_store (a host struct), err_flags
    OUTS = [fake] * 6 + [NULL, fake]
    # bad shapes
    assert f(fake, -1, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, *OUTS, fake, ws, NULL) == -2
    assert f(fake, 4, 0, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, *OUTS, fake, ws, NULL) == -2
    assert f(fake, 4, 10, 9, *[fake] * 4, ctypes.byref(prm), 0, 0, *OUTS, fake, ws, NULL) == -2
    # B == 0 is a no-op
    assert f(NULL, 0, 10, 10, *[NULL] * 4, NULL, 0, 0, *[NULL] * 8, NULL, 0, NULL) == 0
    # required pointers
    assert f(NULL, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, *OUTS, fake, ws, NULL) == -1
    assert f(fake, 4, 10, 10, *[fake] * 4, NULL, 0, 0, *OUTS, fake, ws, NULL) == -1
    # a surprisal store needs both of its arrays
    half = eti.SurpStore(fake, None, 16)
    assert f(fake, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, *[fake] * 6, ctypes.byref(half),
             fake, fake, ws, NULL) == -1
    # workspace
    assert f(fake, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, *OUTS, NULL, ws, NULL) == -4
    assert f(fake, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, *OUTS, fake, ws - 1, NULL) == -4


def test_attention_call_validation(lib):
    P = ctypes.c_void_p
    a16 = P(4096)
    bad = P(4098)
    f = lib.eti_score_prune_blocks
    need = lib.eti_score_prune_workspace_size(4, 32, 8, 128, 16, 512)
    assert need >= 4 * 32 * 512 * 16
    base = dict(B=4, Hq=32, Hkv=8, D=128, P=16, mb=512)

    def call(q=a16, k=a16, B=4, Hq=32, Hkv=8, D=128, Pg=16, mb=512, ws=a16, wsb=None, mode=0,
             surp=NULL):
        wsb = need if wsb is None else wsb
        return f(q, k, a16, a16, B, Hq, Hkv, D, Pg, mb, 1000, 0.1, a16, 1, mode, surp,
                 a16, a16, a16, NULL, NULL, NULL, a16, ws, wsb, NULL)
    assert call(mode=3) == -3                # unknown score mode
    assert call(mode=-1) == -3
    assert call(mode=1) == -1                # mode E needs the surprisal store
    assert call(Hq=30) == -2                 # Hq % Hkv
    assert call(Hq=72, Hkv=8) == -3          # g > 8
    assert call(D=96) == -3
    assert call(Pg=8) == -3
    assert call(mb=0) == -2
    assert call(mb=40000) == -3
    assert call(B=9000) == -2
    assert call(q=NULL) == -1
    assert call(q=bad) == -6
    assert call(ws=NULL) == -4
    assert call(wsb=need - 1) == -4
    assert call(B=0, ws=NULL) == 0
    # decode: workspace sizes grow when the scores must be recomputed
    with_s = lib.eti_paged_decode_workspace_size(4, 32, 8, 128, 16, 512, 1)
    without = lib.eti_paged_decode_workspace_size(4, 32, 8, 128, 16, 512, 0)
    assert 0 < with_s < without
    g = lib.eti_paged_decode
    assert g(a16, a16, a16, a16, a16, 4, 32, 8, 128, 16, 512, 1000, 0.1,
             NULL, NULL, NULL, NULL, NULL, a16, a16, a16, without - 1, NULL) == -4
    assert g(a16, a16, bad, a16, a16, 4, 32, 8, 128, 16, 512, 1000, 0.1,
             NULL, NULL, NULL, NULL, NULL, a16, a16, a16, without, NULL) == -6


def test_binding_refuses_cpu_tensors(lib):
    import torch
    x = torch.zeros(2, 8)
    with pytest.raises(eti.EtiError):
        eti.eti_entropy_temp_sample(x, x[:, 0], x[:, 0], x[:, 0], x[:, 0],
                                    torch.zeros(2, dtype=torch.int32), x[:, 0], x[:, 0],
                                    torch.zeros(2, dtype=torch.int32), torch.zeros(64, dtype=torch.uint8))
