"""Guard bands around every output and workspace buffer of the step.

Each buffer a call writes is carved out of a larger allocation whose first
and last 4 KB hold a fill pattern; after the whole decode step (scores, keep
set, pruned decode, entropy and sample) the bands must still hold it, and
the results must equal those of the same step on plain buffers.  A kernel
that writes past the extent include/eti.h documents for a buffer (a wrong
stride, a missed tail guard) changes a band even where the parity tests,
whose neighbouring allocations are hundreds of bytes apart, would not see it.
The harness itself is checked on the CPU.
"""
import math

import numpy as np
import pytest
import torch

import workloads

GUARD = 4096          # bytes on each side; a multiple of 256 keeps every alignment
FILL = 0xA5


class Guarded:
    """A tensor of the given shape and dtype inside a guard-banded byte buffer."""

    def __init__(self, shape, dtype, device):
        n = math.prod(shape) * torch.empty((), dtype=dtype).element_size()
        self.buf = torch.full((GUARD + n + GUARD,), FILL, dtype=torch.uint8, device=device)
        self.t = self.buf[GUARD:GUARD + n].view(dtype).view(shape)

    def intact(self) -> bool:
        return bool((self.buf[:GUARD] == FILL).all()) and bool((self.buf[-GUARD:] == FILL).all())


def guard_buffers(obj, names, device):
    """Replace the named tensor attributes of obj by guarded tensors of the
    same shape and dtype; returns {name: Guarded}."""
    out = {}
    for n in names:
        t = getattr(obj, n)
        g = Guarded(tuple(t.shape), t.dtype, device)
        setattr(obj, n, g.t)
        out[n] = g
    return out


def test_harness_detects_a_write_past_either_end():
    class Obj:
        pass
    o = Obj()
    o.a = torch.zeros((3, 5), dtype=torch.float32)
    o.b = torch.zeros(7, dtype=torch.bfloat16)
    gs = guard_buffers(o, ["a", "b"], "cpu")
    assert o.a.shape == (3, 5) and o.a.dtype == torch.float32 and o.a.is_contiguous()
    assert o.a.data_ptr() % 256 == gs["a"].buf.data_ptr() % 256
    o.a.fill_(1.0)                     # every element of the extent: fine
    o.b.fill_(2.0)
    assert all(g.intact() for g in gs.values())
    assert (o.a == 1).all() and (gs["a"].buf[GUARD:GUARD + 60].view(torch.float32) == 1).all()
    gs["a"].buf[GUARD + 60] = 0        # one byte past the end
    assert not gs["a"].intact()
    gs["b"].buf[GUARD - 1] = 0         # one byte before the start
    assert not gs["b"].intact()


STEP_BUFFERS = ("keep_mask", "kept_idx", "kept_cnt", "block_score", "token_scores", "kept_norm",
                "err_attn", "err_dec", "err_ets", "out", "tok", "H", "T_out", "dH", "theta_next",
                "surprisal", "ws_score", "ws_dec", "ws_ets")


def _run_step(eti, w, kv, lg, theta, guarded):
    st = eti.DecodeStep(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, w.V, device="cuda:0")
    gs = guard_buffers(st, STEP_BUFFERS, "cuda:0") if guarded else {}
    st.attention(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                 kv["scale"], theta, 2, num_pages=kv["num_pages"])
    tau = lg["tau"].clone()
    st.sample(lg["logits"], lg["T_in"], lg["H_prev"], tau, lg["H_target"], seed=5, offset=1)
    torch.cuda.synchronize()
    res = {n: getattr(st, n).clone() for n in STEP_BUFFERS if not n.startswith("ws_")}
    res["tau"] = tau
    return res, gs


@pytest.mark.gpu
@pytest.mark.parametrize("case", ["gqa4_d128_p16", "gqa4_d64_p32_edges"])
def test_step_writes_stay_inside_their_buffers(case):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as eti
    eti.build()
    eti.load()
    if case == "gqa4_d128_p16":
        w = workloads.Workload("c1", B=5, Hq=16, Hkv=4, D=128, P=16, V=4099,
                               ctx=("list", [1, 37, 1000, 16, 333]), seed=51, hi_frac=0.1)
    else:
        w = workloads.Workload("c2", B=4, Hq=8, Hkv=2, D=64, P=32, V=1001,
                               ctx=("list", [0, 70, 70, 64]), seed=52)
    kv = workloads.make_kv(w, "cuda:0", poison_tail=True)
    lg = workloads.make_logits(w, "cuda:0")
    if case != "gqa4_d128_p16":
        kv["block_table"][2, 1] = kv["num_pages"] + 7      # a bad page id
        lg["logits"][3, 5] = float("nan")                  # an error row
    theta = torch.full((w.B,), 0.8, dtype=torch.float32, device="cuda:0")
    plain, _ = _run_step(eti, w, kv, lg, theta, guarded=False)
    got, gs = _run_step(eti, w, kv, lg, theta, guarded=True)
    bad = [n for n, g in gs.items() if not g.intact()]
    assert not bad, f"writes outside the buffer extent: {bad}"
    # token scores are defined for the blocks of each sequence (slots past its
    # last block are never written); every other buffer over its whole extent
    L = kv["ctx_lens"].cpu().numpy()
    for n, t in plain.items():
        a, b = t.cpu(), got[n].cpu()
        if n == "token_scores":
            a = torch.cat([a[i, :, :-(-int(L[i]) // w.P)].reshape(-1) for i in range(w.B)])
            b = torch.cat([b[i, :, :-(-int(L[i]) // w.P)].reshape(-1) for i in range(w.B)])
        if a.dtype in (torch.float32, torch.bfloat16):
            assert torch.equal(torch.isnan(a), torch.isnan(b)), n
            a, b = torch.nan_to_num(a.float()), torch.nan_to_num(b.float())
        assert torch.equal(a, b), n
    if case != "gqa4_d128_p16":
        assert got["err_attn"].cpu().tolist()[2] != 0 and got["err_ets"].cpu().tolist()[3] != 0


def _estimator_and_scheduler(eti, lg, B, dev, guarded):
    """eti_topk_entropy and eti_schedule on guarded (or plain) output buffers."""
    f32, i32, u8 = torch.float32, torch.int32, torch.uint8
    spec = {"H_tilde": f32, "H_hat": f32, "tail_mass": f32, "err": i32, "priority": f32,
            "admit": u8, "ema": f32}
    gs, t = {}, {}
    for n, dt in spec.items():
        if guarded:
            gs[n] = Guarded((B,), dt, dev)
            t[n] = gs[n].t
        else:
            t[n] = torch.empty(B, dtype=dt, device=dev)
    t["ema"].copy_(torch.linspace(0.0, 0.5, B, device=dev))
    _topk(eti, lg, t)
    _sched(eti, lg, t, B, dev)
    torch.cuda.synchronize()
    return {n: v.clone() for n, v in t.items()}, gs


def _topk(eti, lg, t):
    eti.eti_topk_entropy(lg["logits"], lg["T_in"], 64, t["H_tilde"], t["H_hat"], t["err"],
                         tail_mass=t["tail_mass"])


def _sched(eti, lg, t, B, dev):
    dH = (lg["H_prev"] - 1.0).contiguous()
    kept = (torch.arange(B * 4, device=dev) % 50).to(torch.int32).view(B, 4)
    ctx = (torch.arange(B, device=dev) * 37 % 4000).to(torch.int32)
    urg = torch.ones(B, dtype=torch.float32, device=dev)
    eti.eti_schedule(dH, t["ema"], B // 2, t["priority"], t["admit"], kept_cnt=kept, P=16,
                     ctx_lens=ctx, urgency=urg)


def test_estimator_and_scheduler_calls_reach_the_device_check():
    # the calls the GPU test below makes are well formed: with host tensors
    # they get as far as the binding's device check
    import paper_2603_03310_gb300 as eti
    w = workloads.WORKLOADS["llama3_8b"].scaled(B=5, V=300)
    lg = workloads.make_logits(w, "cpu")
    t = {n: Guarded((w.B,), dt, "cpu").t for n, dt in
         (("H_tilde", torch.float32), ("H_hat", torch.float32), ("tail_mass", torch.float32),
          ("err", torch.int32), ("priority", torch.float32), ("admit", torch.uint8),
          ("ema", torch.float32))}
    with pytest.raises(eti.EtiError, match="CUDA tensor"):
        _topk(eti, lg, t)
    with pytest.raises(eti.EtiError, match="CUDA tensor"):
        _sched(eti, lg, t, w.B, "cpu")


@pytest.mark.gpu
def test_estimator_and_scheduler_writes_stay_inside_their_buffers():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as eti
    eti.build()
    eti.load()
    w = workloads.WORKLOADS["llama3_8b"].scaled(B=37, V=5003)
    lg = workloads.make_logits(w, "cuda:0")
    lg["logits"][4, 7] = float("nan")                      # an error row
    plain, _ = _estimator_and_scheduler(eti, lg, w.B, "cuda:0", guarded=False)
    got, gs = _estimator_and_scheduler(eti, lg, w.B, "cuda:0", guarded=True)
    bad = [n for n, g in gs.items() if not g.intact()]
    assert not bad, f"writes outside the buffer extent: {bad}"
    for n, a in plain.items():
        a, b = a.cpu(), got[n].cpu()
        if a.dtype == torch.float32:
            assert torch.equal(torch.isnan(a), torch.isnan(b)), n
            a, b = torch.nan_to_num(a), torch.nan_to_num(b)
        assert torch.equal(a, b), n
    assert got["err"].cpu().tolist()[4] != 0
