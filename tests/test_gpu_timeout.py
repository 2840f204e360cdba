"""The failure path of the device-side waits, driven without any GPU hazard.

A wait for a tile copy that gives up marks the blocks its warp did not finish
(NaN block stats from the scoring pass; the decode pass flags its segments),
the keep-set pass turns NaN stats into ETI_ERRF_TIMEOUT with nothing kept,
and the decode writes zeros for what it could not finish.  Two ways in:
  (a) block stats with NaN rows made on the host and fed to eti_prune_blocks:
      exactly what the scorer writes after a timed-out copy (with l - 1 = +inf
      when the drain of the copies in flight gave up too: ETI_ERRF_DRAIN);
  (b) eti_set_wait_limit(0): every tile wait gives up at once, while the
      copies already issued are still drained with the default limit, so no
      copy is left in flight; afterwards the default limit gives the normal
      results again in the same context.
"""
import numpy as np
import pytest
import torch

import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
TIMEOUT, DRAIN = 0x20, 0x40


@pytest.fixture(scope="module")
def eti():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as m
    m.build()
    m.load()
    yield m
    m.set_wait_limit(-1)


def _bufs(w):
    g = w.Hq // w.Hkv
    i32, f32, u8 = torch.int32, torch.float32, torch.uint8
    return dict(stats=torch.empty((w.B, w.Hkv, w.max_blocks, g, 4), dtype=f32, device=DEV),
                scores=torch.empty((w.B, w.Hkv, w.max_blocks, w.P, g), dtype=f32, device=DEV),
                mask=torch.empty((w.B, w.Hkv, w.max_blocks), dtype=u8, device=DEV),
                kidx=torch.empty((w.B, w.Hkv, w.max_blocks), dtype=i32, device=DEV),
                kcnt=torch.empty((w.B, w.Hkv), dtype=i32, device=DEV),
                norm=torch.empty((w.B, w.Hq, 2), dtype=f32, device=DEV),
                err_a=torch.empty(w.B, dtype=i32, device=DEV),
                err_d=torch.empty(w.B, dtype=i32, device=DEV),
                out=torch.empty((w.B, w.Hq, w.D), dtype=torch.bfloat16, device=DEV))


def _score(eti, w, kv, o):
    eti.eti_score_blocks(kv["q"], kv["k_cache"], kv["block_table"], kv["ctx_lens"], kv["scale"],
                         o["stats"], token_scores=o["scores"], num_pages=kv["num_pages"])


def _prune(eti, w, kv, o, theta, B_min=1):
    shape = (w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks)
    eti.eti_prune_blocks(o["stats"], kv["block_table"], kv["ctx_lens"], shape, theta, B_min, o["mask"],
                         o["kidx"], o["kcnt"], o["err_a"], kept_norm=o["norm"], num_pages=kv["num_pages"])


def _decode(eti, w, kv, o):
    ws = torch.empty(eti.paged_decode_workspace_size(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, True),
                     dtype=torch.uint8, device=DEV)
    eti.eti_paged_decode(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                         kv["scale"], o["out"], o["err_d"], ws, kept_idx=o["kidx"], kept_cnt=o["kcnt"],
                         token_scores=o["scores"], kept_norm=o["norm"], num_pages=kv["num_pages"])


def _workload(long_segments):
    # the tile keep-set kernel (max_blocks * g <= 8192) or the wide one
    lens = [3000, 700, 1, 2500, 0] if not long_segments else [40000, 65536, 9000]
    return workloads.Workload("t", B=len(lens), Hq=32, Hkv=8, D=128, P=16, V=16, ctx=("list", lens),
                              seed=5, hi_frac=0.05)


@pytest.mark.parametrize("long_segments", [False, True])
def test_nan_stats_report_timeout(eti, long_segments):
    """(a): NaN block stats (a scoring pass that gave up) -> ETI_ERRF_TIMEOUT,
    nothing kept, zero decode output for those segments; +inf in l - 1 adds
    ETI_ERRF_DRAIN; every other segment is unchanged."""
    w = _workload(long_segments)
    kv = workloads.make_kv(w, DEV)
    theta = torch.full((w.B,), 0.8, device=DEV)
    clean = _bufs(w)
    _score(eti, w, kv, clean)
    _prune(eti, w, kv, clean, theta)
    _decode(eti, w, kv, clean)
    bad = _bufs(w)
    _score(eti, w, kv, bad)
    nan = float("nan")
    # sequence 0: blocks from 5 on of every kv head, as a warp that gave up mid-sequence
    bad["stats"][0, :, 5:, :, 0] = nan
    bad["stats"][0, :, 5:, :, 1] = nan
    bad["stats"][0, :, 5:, :, 2] = nan
    # sequence 1: kv head 3 only, with the drain mark
    bad["stats"][1, 3, 2:, :, 0] = nan
    bad["stats"][1, 3, 2:, :, 1] = float("inf")
    _prune(eti, w, kv, bad, theta)
    _decode(eti, w, kv, bad)
    torch.cuda.synchronize()
    err = bad["err_a"].cpu().numpy().view(np.uint32)
    assert err[0] == TIMEOUT
    assert err[1] == TIMEOUT | DRAIN
    assert (err[2:] == clean["err_a"].cpu().numpy().view(np.uint32)[2:]).all()
    cnt, cnt0 = bad["kcnt"].cpu().numpy(), clean["kcnt"].cpu().numpy()
    assert (cnt[0] == 0).all() and cnt[1, 3] == 0
    out, out0 = bad["out"].float().cpu().numpy(), clean["out"].float().cpu().numpy()
    g = w.Hq // w.Hkv
    assert (out[0] == 0).all() and (out[1, 3 * g:4 * g] == 0).all()
    # untouched segments: the same keep sets; the same outputs up to the
    # rounding of the decode's re-split fp32 sums (two bf16 ulps)
    keep = np.ones((w.B, w.Hkv), bool)
    keep[0] = False
    keep[1, 3] = False
    assert (cnt[keep] == cnt0[keep]).all()
    m, m0 = bad["mask"].cpu().numpy(), clean["mask"].cpu().numpy()
    assert np.array_equal(m[keep], m0[keep])
    heads = np.repeat(keep, g, axis=1)
    a, c = out[heads], out0[heads]
    assert np.all(np.abs(a - c) <= 2.0 ** -7 * np.maximum(np.abs(a), np.abs(c)) + 1e-3)


def test_wait_limit_zero_reports_timeout_and_recovers(eti):
    """(b): with a wait limit of 0 every tile wait gives up at once; the copies
    in flight are drained, every sequence with blocks reports ETI_ERRF_TIMEOUT
    (and no DRAIN), nothing is kept, the outputs are zero; the same calls with
    the default limit then match a clean run bit for bit."""
    w = _workload(False)
    kv = workloads.make_kv(w, DEV)
    theta = torch.full((w.B,), 0.8, device=DEV)
    clean = _bufs(w)
    _score(eti, w, kv, clean)
    _prune(eti, w, kv, clean, theta)
    _decode(eti, w, kv, clean)
    torch.cuda.synchronize()
    L = kv["ctx_lens"].cpu().numpy()
    has = L > 0

    prev = eti.set_wait_limit(0)
    try:
        o = _bufs(w)
        _score(eti, w, kv, o)
        _prune(eti, w, kv, o, theta)
        _decode(eti, w, kv, o)
        torch.cuda.synchronize()
    finally:
        eti.set_wait_limit(prev)
    err = o["err_a"].cpu().numpy().view(np.uint32)
    assert (err[has] == TIMEOUT).all() and (err[~has] == 0).all()
    assert (o["kcnt"].cpu().numpy() == 0).all()
    assert (o["out"].float().cpu().numpy() == 0).all()

    # the decode pass alone: keep sets from a normal scoring pass, decode waits give up
    o2 = _bufs(w)
    _score(eti, w, kv, o2)
    _prune(eti, w, kv, o2, theta)
    torch.cuda.synchronize()
    prev = eti.set_wait_limit(0)
    try:
        _decode(eti, w, kv, o2)
        torch.cuda.synchronize()
    finally:
        eti.set_wait_limit(prev)
    errd = o2["err_d"].cpu().numpy().view(np.uint32)
    kept = o2["kcnt"].cpu().numpy().sum(1) > 0
    assert (errd[kept] == TIMEOUT).all() and (errd[~kept] == 0).all()
    assert (o2["out"].float().cpu().numpy() == 0).all()

    # back to the default limit: the same context gives the clean results
    o3 = _bufs(w)
    _score(eti, w, kv, o3)
    _prune(eti, w, kv, o3, theta)
    _decode(eti, w, kv, o3)
    torch.cuda.synchronize()
    for k in ("mask", "kidx", "kcnt", "err_a", "err_d"):
        assert torch.equal(o3[k], clean[k]), k
    assert torch.equal(o3["out"], clean["out"])
