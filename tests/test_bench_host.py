"""Host logic of bench.py that decides what the JSON line reports (CPU only).

The clock summary decides whether a run is kept (a thermal or hardware
slowdown rejects it), the source digest decides whether the committed ncu
traffic still describes the kernel that ran, and the byte accounting is the
numerator of every roofline fraction.  None of this needs a GPU.
"""
import json
import os

import numpy as np
import pytest

import bench
import workloads


def _line(sm, mx=2070, reasons=("Not Active",) * 4, power=900.0):
    hw, hwt, swt, cap = reasons
    return f"0, {sm}, {mx}, {power}, 0x0000000000000000, {hw}, {hwt}, {swt}, {cap}"


def test_clock_summary_median_max_and_reasons():
    c = bench.ClockSampler(0)
    c.lines = [_line(2070), _line(1995), _line(2070),
               _line(1900, reasons=("Not Active", "Not Active", "Not Active", "Active")),
               "garbage", "0, [N/A], 2070, 1.0, 0x0, Not Active, Not Active, Not Active, Not Active"]
    s = c.summary()
    assert s["sm_mhz"] == 2032.5 and s["sm_max_mhz"] == 2070.0 and s["samples"] == 4
    assert s["reasons"] == ["sw_power_cap"]
    c.lines = [_line(1200, reasons=("Active", "Not Active", "Active", "Not Active"))]
    assert c.summary()["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    c.lines = []
    assert c.summary() is None


def test_clock_sampler_without_nvidia_smi(monkeypatch, tmp_path):
    # no nvidia-smi on the host: the sampler is a no-op and reports nothing
    monkeypatch.setenv("PATH", str(tmp_path))
    log = tmp_path / "clocks.csv"
    with bench.ClockSampler(0, str(log)) as c:
        pass
    assert c.summary() is None and not log.exists()


def test_source_digest_ignores_comments_not_code(tmp_path):
    a = tmp_path / "a.cu"
    a.write_text("int f(int x) {\n    return x + 1;  // add one\n}\n")
    d0 = bench.source_digest([str(a)])
    a.write_text("/* header */\n\nint f(int x) {\n    return x + 1;  // plus one\n}\n")
    assert bench.source_digest([str(a)]) == d0
    a.write_text("int f(int x) {\n    return x + 2;\n}\n")
    assert bench.source_digest([str(a)]) != d0


def test_ncu_traffic_record_matches_the_committed_kernels():
    rec = json.load(open(os.path.join(bench.ROOT, "profiles", "ncu_traffic.json")))
    kernels = [k for k in rec if not k.startswith("_")]
    assert {"score_blocks", "paged_decode", "entropy_sample", "prune_finalize"} <= set(kernels)
    for k in kernels:
        for p in rec[k]["sources"]:
            assert os.path.exists(os.path.join(bench.ROOT, p)), p
        got = bench.ncu_traffic(k)
        # a record is either current (its bytes) or stale (None), never wrong
        assert got in (rec[k]["bytes"], None)
    assert bench.ncu_traffic("no_such_kernel") is None


def test_algorithmic_bytes_of_the_step():
    w = workloads.WORKLOADS["llama3_8b"]
    L = workloads.ctx_lengths(w)
    nb = -(-L // w.P)
    g = w.Hq // w.Hkv
    kept = int(nb.sum()) * w.Hkv // 2
    b = bench.algorithmic_bytes(w, L, kept)
    # every key of every sequence once (bf16), per kv head
    keys = sum(int(l) * w.Hkv * w.D * 2 for l in L)
    assert b["score"] > keys and b["score"] - keys < 0.25 * keys      # + q, scores, stats
    # the decode reads only the kept V pages (and their scores): half kept,
    # about half of all V
    allv = sum(int(n) * w.P * w.Hkv * (w.D * 2 + g * 4) for n in nb)
    assert abs(b["decode"] - allv / 2) < w.B * w.Hq * w.D * 2 + 1
    assert b["sample"] == w.B * w.V * 4
    assert 0 < b["prune"] < b["score"] / 10
    # the keep-all decode bytes scale linearly with the kept blocks
    b2 = bench.algorithmic_bytes(w, L, 2 * kept)
    assert b2["decode"] - b["decode"] == b["decode"] - bench.algorithmic_bytes(w, L, 0)["decode"]


def test_aggregate_counts_every_rank_over_the_slowest():
    v, slow = bench.aggregate([0.010, 0.012, 0.011, 0.009], 64)
    assert slow == 0.012 and v == pytest.approx(4 * 64 / 0.012)
    assert bench.max_over_ranks(3.5, 1, None) == 3.5


def test_shards_are_independent_batches_of_the_same_shape():
    w = workloads.WORKLOADS["llama3_8b"]
    shards = [bench.shard_workload(w, r) for r in range(4)]
    assert shards[0] == w
    assert len({s.seed for s in shards}) == 4
    assert all((s.B, s.Hq, s.Hkv, s.D, s.P, s.V, s.ctx) == (w.B, w.Hq, w.Hkv, w.D, w.P, w.V, w.ctx)
               for s in shards)
    Ls = [workloads.ctx_lengths(s) for s in shards]
    assert not np.array_equal(Ls[0], Ls[1])


def test_warmup_is_at_least_three(monkeypatch):
    seen = {}
    monkeypatch.setattr(bench, "run_gpu", lambda a: seen.update(gpu=a))
    monkeypatch.setattr(bench, "run_reference", lambda a: seen.update(ref=a))
    bench.main(["--steps", "5", "--warmup", "1"])
    assert seen["gpu"].warmup == 3 and seen["gpu"].steps == 5
    bench.main(["--impl", "reference", "--steps", "2", "--warmup", "0"])
    assert seen["ref"].impl == "reference" and seen["ref"].warmup == 0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    # under torchrun the other ranks exit without work and print nothing
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    import argparse
    args = argparse.Namespace(workload="tiny", steps=3, warmup=3, cpu_budget=1.0)
    assert bench.run_reference(args) is None
    assert capsys.readouterr().out == ""


def test_reference_arm_line_on_the_tiny_step(monkeypatch, capsys, oracle_lib):
    monkeypatch.setenv("RANK", "0")
    monkeypatch.setenv("WORLD_SIZE", "1")
    bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "3", "--warmup", "3",
                "--cpu-budget", "2"])
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["value"] > 0 and line["unit"] == bench.UNIT and line["higher_is_better"] is True
    assert line["config"]["workload"] == bench.workload_desc(workloads.WORKLOADS["tiny"])
    assert line["config"]["workload"].startswith("tiny: B=4 Hq=8 Hkv=8 D=64 P=16")
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": bench.UNIT, "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


def test_e2e_working_set_exceeds_l2():
    # the end-to-end leg runs without an L2 flush: the keys alone that a step
    # of the benchmark workload reads are several times the 129 MB L2
    import torch
    w = workloads.WORKLOADS["llama3_8b"]
    L = workloads.ctx_lengths(w)
    kb = bench.key_bytes(w, {"ctx_lens": torch.from_numpy(L)})
    assert kb >= int(L.sum()) * w.Hkv * w.D * 2
    assert kb > 4 * 129 * 2 ** 20


def test_e2e_at_one_rank_is_reported_as_measured():
    e = {"value": 123.0, "unit": "tokens/s", "ms_per_step": 0.5, "h2d_bytes_per_step": 9,
         "d2h_bytes_per_step": 3, "mode": "x"}
    assert bench.aggregate_e2e(e, 64, 1, None) is e


def test_kept_attention_mass_matches_the_oracle(oracle_lib):
    # block stats in the scorer's layout, formed in fp64 from the same bf16
    # inputs; the oracle's per-block attention masses summed over its keep set
    # give the expected share for every query head
    import math
    import torch
    oracle = oracle_lib
    w = workloads.Workload("km", B=4, Hq=8, Hkv=2, D=64, P=16, V=16,
                           ctx=("list", [37, 0, 200, 16]), seed=71, hi_frac=0.2)
    kv = workloads.make_kv(w, "cpu")
    g, mb = w.Hq // w.Hkv, w.max_blocks
    qb, kb = workloads.bf16_bits(kv["q"]), workloads.bf16_bits(kv["k_cache"])
    bt, L = kv["block_table"].numpy(), kv["ctx_lens"].numpy()
    ref = oracle.score_prune(qb, kb, bt, L, kv["scale"], np.full(w.B, 0.9), 2, want_heads=True)
    q = kv["q"].double()
    stats = torch.full((w.B, w.Hkv, mb, g, 4), float("nan"), dtype=torch.float32)  # unwritten
    for b in range(w.B):
        nb = -(-int(L[b]) // w.P)
        for j in range(nb):
            n = min(w.P, int(L[b]) - j * w.P)
            k = kv["k_cache"][int(bt[b, j])].double()[:, :n]            # [Hkv, n, D]
            for h in range(w.Hq):
                x = (k[h // g] @ q[b, h]) * kv["scale"]
                m = x.max()
                stats[b, h // g, j, h % g, 0] = float(m)
                stats[b, h // g, j, h % g, 1] = float(torch.exp(x - m).sum() - 1.0)
    keep = torch.from_numpy(ref["keep_mask"])
    got = bench.kept_attention_mass(stats, keep, kv["ctx_lens"], w.P)
    want = []
    for b in range(w.B):
        if L[b] == 0:
            continue
        for h in range(w.Hq):
            kept = ref["keep_mask"][b, h // g].astype(bool)
            want.append(ref["head_A"][b, h][kept].sum())
    assert got["mean"] == pytest.approx(float(np.mean(want)), abs=2e-5)
    assert got["min"] == pytest.approx(float(np.min(want)), abs=2e-5)
    assert 0 < got["min"] <= got["mean"] <= 1
    # keeping every block keeps all of the attention
    full = bench.kept_attention_mass(stats, torch.ones_like(keep), kv["ctx_lens"], w.P)
    assert full["mean"] == pytest.approx(1.0, abs=1e-6) and full["min"] == pytest.approx(1.0, abs=1e-6)


def test_sub_batches_cover_the_batch_in_order():
    """The overlapped step's sub-batches: contiguous, in order, disjoint,
    covering every sequence once, none empty, sizes within one of each other."""
    for B in (1, 2, 3, 4, 7, 8, 64, 65, 128, 256, 8191):
        for n in (1, 2, 3, 4, 8):
            runs = bench.sub_batches(B, n)
            assert len(runs) == min(n, B)
            assert runs[0][0] == 0 and runs[-1][1] == B
            assert all(a[1] == b[0] for a, b in zip(runs, runs[1:]))
            sizes = [hi - lo for lo, hi in runs]
            assert min(sizes) >= 1 and max(sizes) - min(sizes) <= 1


def test_sub_batches_by_weight_balance_the_work():
    """With per-sequence weights the cuts fall where the running weight
    crosses each share of the total (the best cut in the sequence order),
    the runs stay contiguous and non-empty."""
    rng = np.random.default_rng(0)
    for B in (2, 3, 7, 64, 256):
        wts = rng.integers(1, 512, size=B)
        for n in (1, 2, 3, 4):
            runs = bench.sub_batches(B, n, weights=wts)
            assert len(runs) == min(n, B)
            assert runs[0][0] == 0 and runs[-1][1] == B
            assert all(a[1] == b[0] and a[0] < a[1] for a, b in zip(runs, runs[1:]))
            if n == 2 and B > 2:
                cut = runs[0][1]
                tot = wts.sum()
                best = min(abs(wts[:k].sum() - tot / 2) for k in range(1, B))
                assert abs(wts[:cut].sum() - tot / 2) == best
    assert bench.sub_batches(4, 2, weights=[1, 1, 1, 100]) == [(0, 3), (3, 4)]
    assert bench.sub_batches(4, 2, weights=[100, 1, 1, 1]) == [(0, 1), (1, 4)]

