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
    for s in (0, -1, -2, -3, -4, -5, -6, -7, -8):
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
    assert f(fake, -1, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, fake, ws, NULL) == -2
    assert f(fake, 4, 0, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, fake, ws, NULL) == -2
    assert f(fake, 4, 10, 9, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, fake, ws, NULL) == -2
    # B == 0 is a no-op
    assert f(NULL, 0, 10, 10, *[NULL] * 4, NULL, 0, 0, NULL, *[NULL] * 8, NULL, 0, NULL) == 0
    # required pointers
    assert f(NULL, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, fake, ws, NULL) == -1
    assert f(fake, 4, 10, 10, *[fake] * 4, NULL, 0, 0, NULL, *OUTS, fake, ws, NULL) == -1
    # a surprisal store needs both of its arrays
    half = eti.SurpStore(fake, None, 16)
    assert f(fake, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *[fake] * 6, ctypes.byref(half),
             fake, fake, ws, NULL) == -1
    # workspace
    assert f(fake, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, NULL, ws, NULL) == -4
    assert f(fake, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, fake, ws - 1, NULL) == -4


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
    assert call(q=bad) == -8
    assert call(ws=NULL) == -4
    assert call(wsb=need - 1) == -4
    assert call(B=0, ws=NULL) == 0
    # 32-bit device indices: unit counts B*Hkv*max_blocks and cache rows
    # num_pages*Hkv*P are bounded even where each size alone is allowed
    assert call(B=8192, Hq=32, Hkv=8, mb=32768) == -3
    assert call(B=8192, Hq=32, Hkv=8, mb=16384, q=NULL) == -1   # 2^30 units: accepted
    assert f(a16, a16, a16, a16, 4, 32, 8, 128, 16, 512, (1 << 31) // (8 * 16) + 1, 0.1, a16, 1, 0,
             NULL, a16, a16, a16, NULL, NULL, NULL, a16, a16, need, NULL) == -3
    assert f(a16, a16, a16, a16, 4, 32, 8, 128, 16, 512, (1 << 31) // (8 * 16) - 1, 0.1, a16, 1, 0,
             NULL, a16, a16, a16, NULL, NULL, NULL, a16, NULL, need, NULL) == -4
    assert lib.eti_score_prune_workspace_size(8192, 32, 8, 128, 16, 32768) == 0
    # decode: workspace sizes grow when the scores must be recomputed
    with_s = lib.eti_paged_decode_workspace_size(4, 32, 8, 128, 16, 512, 1)
    without = lib.eti_paged_decode_workspace_size(4, 32, 8, 128, 16, 512, 0)
    assert 0 < with_s < without
    g = lib.eti_paged_decode
    assert g(a16, a16, a16, a16, a16, 4, 32, 8, 128, 16, 512, 1000, 0.1,
             NULL, NULL, NULL, NULL, NULL, a16, a16, a16, without - 1, NULL) == -4
    assert g(a16, a16, bad, a16, a16, 4, 32, 8, 128, 16, 512, 1000, 0.1,
             NULL, NULL, NULL, NULL, NULL, a16, a16, a16, without, NULL) == -8


def test_binding_refuses_cpu_tensors(lib):
    import torch
    x = torch.zeros(2, 8)
    with pytest.raises(eti.EtiError):
        eti.eti_entropy_temp_sample(x, x[:, 0], x[:, 0], x[:, 0], x[:, 0],
                                    torch.zeros(2, dtype=torch.int32), x[:, 0], x[:, 0],
                                    torch.zeros(2, dtype=torch.int32), torch.zeros(64, dtype=torch.uint8))


def test_status_strings_cover_every_code(lib):
    for s in (-7,):
        assert "scratch" in lib.eti_status_string(s).decode()
    assert "aligned" in lib.eti_status_string(-8).decode()
    assert "wait" in lib.eti_status_string(-6).decode()


def test_wait_limit_setting(lib):
    # the diagnostic wait limit: set, read back through the previous value, restore
    prev = eti.set_wait_limit(0)
    assert prev == 1 << 20
    assert eti.set_wait_limit(5) == 0
    assert eti.set_wait_limit(-1) == 5
    assert eti.set_wait_limit(-1) == 1 << 20
    assert lib.eti_status_string(-99).decode() == "unknown status"


def test_topk_call_validation(lib):
    P = ctypes.c_void_p
    fake = P(256)
    f = lib.eti_topk_entropy

    def call(logits=fake, B=4, V=10, ld=10, T=fake, k=3, Ht=fake, Hh=fake, tail=fake, err=fake):
        return f(logits, B, V, ld, T, k, Ht, Hh, tail, err, NULL)
    assert call(B=-1) == -2
    assert call(B=65536) == -2
    assert call(V=0) == -2
    assert call(ld=9) == -2                  # rows overlap
    assert call(k=0) == -2
    assert call(B=0, logits=NULL, T=NULL, Ht=NULL, Hh=NULL, err=NULL) == 0
    for name in ("logits", "T", "Ht", "Hh", "err"):
        assert call(**{name: NULL}) == -1, name


def test_schedule_call_validation(lib):
    P = ctypes.c_void_p
    fake = P(256)
    prm = eti.sched_params()
    f = lib.eti_schedule

    def call(dH=fake, ema=fake, kept=NULL, Hkv=8, Pg=16, L=NULL, urg=NULL, p=ctypes.byref(prm),
             B=4, budget=2, pri=fake, adm=fake):
        return f(dH, ema, kept, Hkv, Pg, L, urg, p, B, budget, pri, adm, NULL)
    assert call(B=-1) == -2
    assert call(B=65536) == -2
    assert call(kept=fake, Hkv=0) == -2      # kept counts need the kv-head count
    assert call(kept=fake, Pg=0) == -2       # ... and the page size
    assert call(B=0, dH=NULL, ema=NULL, p=NULL, pri=NULL, adm=NULL) == 0
    for name in ("dH", "ema", "p", "pri", "adm"):
        assert call(**{name: NULL}) == -1, name


def test_score_and_prune_call_validation(lib):
    P = ctypes.c_void_p
    a16, bad = P(4096), P(4100)

    def score(q=a16, k=a16, bt=a16, L=a16, B=4, Hq=32, Hkv=8, D=128, Pg=16, mb=512, pages=1000,
              stats=a16):
        return lib.eti_score_blocks(q, k, bt, L, B, Hq, Hkv, D, Pg, mb, pages, 0.1, NULL, NULL,
                                    stats, NULL)
    assert score(B=-1) == -2
    assert score(pages=-1) == -2
    assert score(Hq=12, Hkv=8) == -2
    assert score(D=256) == -3
    assert score(B=0, q=NULL, k=NULL, bt=NULL, L=NULL, stats=NULL) == 0
    for name in ("q", "k", "bt", "L", "stats"):
        assert score(**{name: NULL}) == -1, name
    for name in ("q", "k", "stats"):
        assert score(**{name: bad}) == -8, name

    def prune(stats=a16, bt=a16, L=a16, B=4, Hq=32, Hkv=8, D=128, Pg=16, mb=512, pages=1000,
              theta=a16, mode=0, mask=a16, kidx=a16, kcnt=a16, err=a16):
        return lib.eti_prune_blocks(stats, bt, L, B, Hq, Hkv, D, Pg, mb, pages, theta, 1, mode,
                                    mask, kidx, kcnt, NULL, NULL, err, NULL)
    assert prune(mb=0) == -2
    assert prune(mb=40000) == -3
    assert prune(Pg=64) == -3
    assert prune(mode=3) == -3
    assert prune(B=0, stats=NULL, bt=NULL, L=NULL, theta=NULL, mask=NULL, kidx=NULL, kcnt=NULL,
                 err=NULL) == 0
    for name in ("stats", "bt", "L", "theta", "mask", "kidx", "kcnt", "err"):
        assert prune(**{name: NULL}) == -1, name
    assert prune(stats=bad) == -8


def test_noalloc_call_validation(lib):
    # every refusal below comes before the library looks up its scratch
    # array on a device, so it runs without a GPU
    P = ctypes.c_void_p
    fake = P(256)
    prm = eti.ctrl_params()
    f = lib.eti_entropy_temp_sample_noalloc
    OUTS = [fake] * 6 + [NULL, fake]
    assert f(fake, -1, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, NULL) == -2
    assert f(fake, 4, 10, 9, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, NULL) == -2
    assert f(NULL, 0, 10, 10, *[NULL] * 4, NULL, 0, 0, NULL, *[NULL] * 8, NULL) == 0
    assert f(NULL, 4, 10, 10, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, NULL) == -1
    assert f(fake, 4, 10, 10, *[fake] * 4, NULL, 0, 0, NULL, *OUTS, NULL) == -1
    # the largest batch whose scratch fits is accepted by the size check; one
    # more row than the array holds is refused with ETI_ERR_TOO_LARGE
    cap = lib.eti_entropy_temp_sample_noalloc_max_bytes()
    lo, hi = 1, 65535
    if lib.eti_entropy_temp_sample_workspace_size(hi, 4) <= cap:
        pytest.skip("every batch fits the fixed scratch on this device")
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if lib.eti_entropy_temp_sample_workspace_size(mid, 4) <= cap:
            lo = mid
        else:
            hi = mid
    assert f(fake, hi, 4, 4, *[fake] * 4, ctypes.byref(prm), 0, 0, NULL, *OUTS, NULL) == -7


def test_binding_constants_match_the_header():
    txt = open(os.path.join(ROOT, "include", "eti.h")).read()
    for name, val in re.findall(r"#define ETI_(ERRF_\w+)\s+(0x[0-9a-fA-F]+)u", txt):
        assert getattr(eti, name) == int(val, 16), name
    for name, val in re.findall(r"#define ETI_(OK|ERR_\w+)\s+\(?(-?\d+)\)?", txt):
        assert int(val) in eti.STATUS, name


C_CLIENT = r"""
#include <math.h>
#include <stdio.h>
#include <string.h>
#include "eti.h"

int main(void) {
    eti_ctrl_params p;
    eti_sched_params s;
    eti_ctrl_defaults(&p);
    eti_sched_defaults(&s);
    if (p.sign != -1.0f || !isinf(p.theta_user) || s.lambda != 0.9f) return 2;
    if (strstr(eti_version(), "libeti") == NULL) return 3;
    if (eti_status_string(ETI_ERR_TOO_LARGE)[0] == 0) return 4;
    if (eti_score_prune_workspace_size(4, 32, 8, 128, 16, 512) == 0) return 5;
    if (eti_score_prune_workspace_size(4, 30, 8, 128, 16, 512) != 0) return 6;
    /* an argument error is reported before anything is enqueued */
    if (eti_entropy_temp_sample(NULL, 4, 10, 10, NULL, NULL, NULL, NULL, &p, 0, 0, NULL, NULL,
                                NULL, NULL, NULL, NULL, NULL, NULL, NULL, NULL, 0, NULL) != ETI_ERR_NULL)
        return 7;
    if (eti_set_wait_limit(-1) != eti_set_wait_limit(-1))
        return 7;
    printf("ok %s\n", eti_version());
    return 0;
}
"""


def test_header_is_plain_c_and_links(lib, tmp_path):
    import shutil, subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    libdir = os.path.dirname(eti.LIB_PATH)
    p = subprocess.run([cc, "-std=c99", "-Wall", "-Werror", "-pedantic", str(src),
                        "-I", os.path.join(ROOT, "include"), "-L", libdir, "-l:libeti.so",
                        "-Wl,-rpath," + libdir, "-lm", "-o", str(exe)],
                       capture_output=True, text=True)
    assert p.returncode == 0, p.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.startswith("ok libeti"), (r.returncode, r.stdout, r.stderr)


def test_readme_c_example_compiles(tmp_path):
    # the decode-step example in the README is compiled against include/eti.h
    import shutil, subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    txt = open(os.path.join(ROOT, "README.md")).read()
    blocks = re.findall(r"```c\n(.*?)```", txt, flags=re.S)
    assert len(blocks) == 1 and "decode_step" in blocks[0]
    src = tmp_path / "example.c"
    src.write_text(blocks[0])
    p = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-c", str(src),
                        "-I", os.path.join(ROOT, "include"), "-o", str(tmp_path / "example.o")],
                       capture_output=True, text=True)
    assert p.returncode == 0, p.stderr
