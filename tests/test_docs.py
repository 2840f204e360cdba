"""The file map and the profiles the design notes cite exist (CPU only)."""
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _design():
    return open(os.path.join(ROOT, "DESIGN.md")).read()


def test_every_cited_repository_path_exists():
    txt = _design() + open(os.path.join(ROOT, "README.md")).read()
    paths = set(re.findall(r"`((?:tests|oracle|include|profiles|workloads|paper_2603_03310_gb300|csrc)"
                           r"/[\w./-]+)`", txt))
    assert paths
    for p in sorted(paths):
        full = os.path.join(ROOT, p)
        if p.startswith("csrc/"):
            full = os.path.join(ROOT, "paper_2603_03310_gb300", p)
        assert os.path.exists(full), p


def test_profiles_name_their_command():
    prof = os.path.join(ROOT, "profiles")
    mds = [f for f in os.listdir(prof) if f.endswith((".md", ".txt"))]
    assert mds
    n_ncu = 0
    for f in mds:
        txt = open(os.path.join(prof, f)).read()
        cmds = "\n".join(re.findall(r"```\n(.*?)```", txt, flags=re.S))
        # a command that runs committed files only, and ncu never locks clocks
        assert "bench.py" in cmds or "buildlib.py" in cmds, f
        for line in cmds.replace("\\\n", " ").splitlines():
            if line.strip().startswith("ncu "):
                assert "--clock-control none" in line, (f, line)
                n_ncu += 1
    assert n_ncu >= 3                     # the launch list and the full captures
