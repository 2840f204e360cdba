"""GPU path vs the fp64 oracle, element by element on the same seeded inputs.

Every call goes through the C ABI (libeti) via the thin binding.  Sizes span
many tiles / CTAs with ragged tails; the full-size workloads are checked on
every row for the entropy/sample half and on sampled sequences (gathered
pages) for the attention half, in the launch configuration the benchmark
times (DecodeStep).
"""
import math

import numpy as np
import pytest
import torch

import oracle
import parity
import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module")
def eti():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as m
    m.build()
    m.load()
    oracle.build()
    return m


def _ctrl_pair(eti, **kw):
    return eti.ctrl_params(**kw), oracle.ctrl(**kw)


# ---------------------------------------------------------------------------
# half (a): entropy, entropic time, temperature, threshold, sample

@pytest.mark.parametrize("name", ["tiny", "llama3_8b", "long_ctx", "mixed_batch", "llama3_70b"])
def test_entropy_sample_full_workloads(eti, name):
    w = workloads.WORKLOADS[name]
    lg = workloads.make_logits(w, DEV)
    fracs = (0.1, 0.3, 0.5) if name == "llama3_70b" else (w.H_target_frac,)
    for f in fracs:
        lg["H_target"].fill_(f * math.log(w.V))
        g = parity.run_ets(eti, lg, seed=w.seed, offset=7)
        r = parity.oracle_ets(lg, seed=w.seed, offset=7)
        st = parity.compare_ets(g, r, lg, seed=w.seed, offset=7)
        print(name, f, st)


@pytest.mark.parametrize("B,V", [(1, 1), (3, 2), (5, 7), (2, 4097), (33, 1000), (7, 50001)])
def test_entropy_sample_ragged_shapes(eti, B, V):
    w = workloads.Workload("r", B=B, Hq=1, Hkv=1, D=64, P=16, V=V, ctx=("list", [1] * B), seed=V)
    lg = workloads.make_logits(w, DEV)
    for seed, off in ((0, 0), (2 ** 40 + 3, 2 ** 33 + 5)):
        g = parity.run_ets(eti, lg, seed=seed, offset=off)
        r = parity.oracle_ets(lg, seed=seed, offset=off)
        parity.compare_ets(g, r, lg, seed=seed, offset=off)


def test_entropy_sample_strided_and_unaligned_rows(eti):
    """ld > V (padded rows) and a base pointer off the 16-byte grid take the scalar path."""
    w = workloads.Workload("s", B=6, Hq=1, Hkv=1, D=64, P=16, V=3001, ctx=("list", [1] * 6), seed=3)
    lg = workloads.make_logits(w, DEV, ld=3008)
    g = parity.run_ets(eti, lg, seed=1, offset=2, V=3001)
    r = parity.oracle_ets(lg, seed=1, offset=2, V=3001)
    parity.compare_ets(g, r, lg, seed=1, offset=2, V=3001)
    # unaligned: view starting one element in
    base = torch.empty(6 * 3001 + 1, dtype=torch.float32, device=DEV)
    base[1:] = lg["logits"][:, :3001].reshape(-1)
    lg2 = dict(lg, logits=base[1:].view(6, 3001))
    g = parity.run_ets(eti, lg2, seed=1, offset=2)
    r = parity.oracle_ets(lg2, seed=1, offset=2)
    parity.compare_ets(g, r, lg2, seed=1, offset=2)


@pytest.mark.parametrize("B,V", [(65535, 37), (2, 1000003)])
def test_entropy_sample_maximum_sizes(eti, B, V):
    """The largest batch the call accepts (65535 rows, a ragged vocabulary) and
    a vocabulary of a million tokens: every row against the oracle."""
    w = workloads.Workload("x", B=B, Hq=1, Hkv=1, D=64, P=16, V=V, ctx=("list", [1] * B), seed=B + V)
    lg = workloads.make_logits(w, DEV)
    g = parity.run_ets(eti, lg, seed=5, offset=11)
    r = parity.oracle_ets(lg, seed=5, offset=11)
    st = parity.compare_ets(g, r, lg, seed=5, offset=11)
    print(B, V, st)


@pytest.mark.parametrize("kw", [dict(), dict(sign=1.0), dict(eta=0.5, T_min=0.5, T_max=1.5),
                                dict(eps_H=0.7, H_min=3.0, theta_user=0.4, theta_hi=2.0),
                                dict(T_cal=1.5), dict(T_cal=0.7, eta=0.3),
                                dict(rho_T=0.05, eta=2.0, T_min=1e-3, T_max=1e3)])
def test_entropy_sample_controller_params(eti, kw):
    w = workloads.WORKLOADS["tiny"].scaled(B=16, ctx=("list", [1] * 16), seed=11)
    lg = workloads.make_logits(w, DEV)
    lg["T_in"].uniform_(0.3, 3.0)
    p, c = _ctrl_pair(eti, **kw)
    g = parity.run_ets(eti, lg, params=p, seed=5, offset=1)
    r = parity.oracle_ets(lg, ctrl=c, seed=5, offset=1)
    parity.compare_ets(g, r, lg, seed=5, offset=1)


def test_entropy_sample_threshold_rate_limit(eti):
    """The dtheta guard: theta_next is read as the previous threshold and the
    new one stays within dtheta of it (non-finite previous values unbounded)."""
    w = workloads.WORKLOADS["tiny"].scaled(B=16, ctx=("list", [1] * 16), seed=12)
    lg = workloads.make_logits(w, DEV)
    base = parity.oracle_ets(lg, seed=3)
    rng = np.random.default_rng(0)
    tp = (base["theta_next"] + rng.uniform(-0.1, 0.1, w.B)).astype(np.float32)
    tp[[2, 9]] = np.inf
    p, c = _ctrl_pair(eti, dtheta=0.02)
    g = parity.run_ets(eti, lg, params=p, seed=3, theta_prev=tp)
    r = parity.oracle_ets(lg, ctrl=c, seed=3, theta_prev=tp)
    parity.compare_ets(g, r, lg, seed=3)
    assert (np.abs(g["theta_next"] - tp)[np.isfinite(tp)] <= 0.02 + 1e-6).all()


def test_entropy_sample_error_rows(eti):
    B, V = 6, 777
    z = torch.randn(B, V, device=DEV)
    z[0, 5] = float("nan")
    z[1, 700] = float("inf")
    z[2, :] = float("-inf")
    z[3, ::2] = float("-inf")           # valid: half the vocabulary masked out
    lg = dict(logits=z, T_in=torch.ones(B, device=DEV), H_prev=torch.zeros(B, device=DEV),
              tau=torch.full((B,), 2.0, device=DEV), H_target=torch.ones(B, device=DEV))
    lg["T_in"][4] = 0.0                  # bad temperature
    lg["T_in"][5] = -1.0
    g = parity.run_ets(eti, lg)
    r = parity.oracle_ets(lg)
    assert list(r["err"]) == [4, 4, 8, 0, 16, 16]
    parity.compare_ets(g, r, lg)
    assert g["tok"][3] % 2 == 1          # never a -inf token
    assert (g["T_out"][[0, 1, 2, 4, 5]] == lg["T_in"].cpu().numpy()[[0, 1, 2, 4, 5]]).all()
    assert (g["theta_next"][[0, 1, 2, 4, 5]] == 0).all()


def test_entropy_sample_near_deterministic_rows(eti):
    """+20 spikes (entropy ~1e-3): absolute entropy tolerance and exact tokens."""
    w = workloads.WORKLOADS["mixed_batch"].scaled(B=32, V=128256)
    lg = workloads.make_logits(w, DEV)
    g = parity.run_ets(eti, lg, seed=3)
    r = parity.oracle_ets(lg, seed=3)
    parity.compare_ets(g, r, lg, seed=3)
    assert (r["H"] < 1e-2).sum() >= 4      # rows where the spike dominates exercise the abs. bound


def test_sampler_distribution_on_gpu(eti):
    """Gumbel-max through the kernel: frequencies over many rows follow softmax."""
    from scipy import stats
    V, N = 6, 60000
    z = torch.tensor([0.0, 1.0, -0.5, 2.0, 0.3, 1.5], device=DEV).repeat(N, 1).contiguous()
    T = 0.8
    lg = dict(logits=z, T_in=torch.full((N,), T, device=DEV), H_prev=torch.zeros(N, device=DEV),
              tau=torch.zeros(N, device=DEV), H_target=torch.ones(N, device=DEV))
    g = parity.run_ets(eti, lg, seed=123, offset=0)
    p = torch.softmax(z[0].double().cpu() / float(np.float32(T)), 0).numpy()
    cnt = np.bincount(g["tok"], minlength=V)
    assert stats.chisquare(cnt, N * p).pvalue > 1e-4
    r = parity.oracle_ets(lg, seed=123, offset=0)
    assert np.mean(g["tok"] == r["tok"]) > 0.9999


def test_entropy_sample_reproducible(eti):
    w = workloads.WORKLOADS["llama3_8b"].scaled(B=8)
    lg = workloads.make_logits(w, DEV)
    a = parity.run_ets(eti, lg, seed=9, offset=4)
    b = parity.run_ets(eti, lg, seed=9, offset=4)
    for k in ("tok", "H", "T_out", "theta_next"):
        assert np.array_equal(a[k], b[k]), k


def _step_ets(st, tau):
    """DecodeStep sampling outputs in the layout parity.compare_ets reads."""
    res = dict(tok=st.tok, H=st.H, T_out=st.T_out, dH=st.dH, theta_next=st.theta_next,
               surprisal=st.surprisal, err=st.err_ets, tau=tau)
    res = {k: v.cpu().numpy() for k, v in res.items()}
    res["err"] = res["err"].view(np.uint32)
    return res


def test_entropy_sample_device_offset(eti):
    """offset_dev: the call reads the Philox offset from a device word and
    leaves it advanced by one, so a captured graph replayed twice draws the
    tokens of two consecutive offsets (each against the oracle)."""
    w = workloads.WORKLOADS["llama3_8b"].scaled(B=16)
    lg = workloads.make_logits(w, DEV)
    st = eti.DecodeStep(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, w.V, device=DEV)
    off = torch.tensor([41], dtype=torch.int64, device=DEV)
    tau = lg["tau"].clone()
    st.sample(lg["logits"], lg["T_in"], lg["H_prev"], tau, lg["H_target"], seed=2, offset=999,
              offset_dev=off)
    torch.cuda.synchronize()
    assert off.item() == 42
    parity.compare_ets(_step_ets(st, tau), parity.oracle_ets(lg, seed=2, offset=41), lg, seed=2, offset=41)
    cs = torch.cuda.Stream(device=DEV)
    cs.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    tau_g = lg["tau"].clone()
    with torch.cuda.graph(graph, stream=cs):
        st.sample(lg["logits"], lg["T_in"], lg["H_prev"], tau_g, lg["H_target"], seed=2, offset_dev=off)
    torch.cuda.synchronize()
    toks = []
    for o in (42, 43):
        tau_g.copy_(lg["tau"])
        graph.replay()
        torch.cuda.synchronize()
        assert off.item() == o + 1
        parity.compare_ets(_step_ets(st, tau_g), parity.oracle_ets(lg, seed=2, offset=o), lg, seed=2,
                           offset=o)
        toks.append(st.tok.clone())
    assert not torch.equal(toks[0], toks[1])


# ---------------------------------------------------------------------------
# half (b): block scores, keep set, pruned paged decode

def _step(eti, w, kv, theta, B_min):
    st = eti.DecodeStep(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, w.V, device=DEV)
    st.attention(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                 kv["scale"], theta, B_min, num_pages=kv["num_pages"])
    torch.cuda.synchronize()
    return st


def _check_step(st, n, theta_np, B_min, P, seqs=None):
    """Compare a DecodeStep's keep set and output with the oracle (on `seqs`)."""
    rng = slice(None) if seqs is None else seqs
    ref = oracle.score_prune(n["q"], n["k"], n["bt"], n["L"], n["scale"], theta_np, B_min,
                             num_pages=n.get("num_pages"), want_heads=True)
    band = parity.score_bands(ref, n)
    gm = st.keep_mask.cpu().numpy()[rng]
    gi = st.kept_idx.cpu().numpy()[rng]
    gc = st.kept_cnt.cpu().numpy()[rng]
    gs = st.block_score.cpu().numpy()[rng]
    worst_s = parity.compare_scores(gs, ref["block_score"], P, n["L"], band)
    mt = parity.compare_masks(gm, gi, gc, ref, theta_np, B_min, P, n["L"], band)
    out_ref, err = oracle.paged_attention(n["q"], n["k"], n["v"], n["bt"], n["L"], n["scale"], gm,
                                          num_pages=n.get("num_pages"))
    worst_o = parity.compare_attention(st.out.float().cpu().numpy()[rng], out_ref)
    assert np.array_equal(st.err_attn.cpu().numpy().view(np.uint32)[rng], ref["err"])
    assert np.array_equal(st.err_dec.cpu().numpy().view(np.uint32)[rng], err)
    return dict(score_err=worst_s, out_err=worst_o, kept=float(gm.sum()), **mt)


SHAPES = [
    # (B, Hq, Hkv, D, P, lens)
    (4, 8, 8, 64, 16, [64, 128, 192, 256]),
    (3, 32, 8, 128, 16, [1, 37, 1000]),
    (5, 16, 2, 128, 32, [33, 64, 500, 17, 2049]),
    (2, 8, 1, 64, 32, [1500, 31]),
    (6, 12, 6, 128, 16, [5, 16, 17, 300, 301, 999]),
    (3, 24, 4, 64, 16, [129, 640, 2]),
    (2, 7, 7, 128, 16, [77, 400]),
    (2, 24, 3, 128, 32, [800, 95]),
    # max_blocks * g of 8192: the keep-set tile kernel with eight warps a segment
    (2, 64, 8, 128, 16, [16384, 5000]),
    (3, 32, 8, 64, 16, [32768, 100, 20000]),
    # 16384 and 32768: clusters of four and eight CTAs a segment (B_min <= 1;
    # larger budgets go to the wide kernel)
    (2, 32, 8, 64, 16, [65536, 3000]),
    (2, 64, 8, 64, 16, [65536, 777]),
]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("theta,B_min", [(0.0, 1), (0.8, 1), (1.0, 3), (float("inf"), 2),
                                         (1.2, 0), (0.5, 10 ** 6)])
def test_score_prune_decode_small(eti, shape, theta, B_min):
    B, Hq, Hkv, D, P, lens = shape
    w = workloads.Workload("p", B=B, Hq=Hq, Hkv=Hkv, D=D, P=P, V=16, ctx=("list", lens),
                           seed=sum(lens) + D + P, hi_frac=0.1)
    kv = workloads.make_kv(w, DEV, poison_tail=True)
    th = torch.full((B,), theta, dtype=torch.float32, device=DEV)
    st = _step(eti, w, kv, th, B_min)
    s = _check_step(st, parity.host_kv(kv), th.cpu().numpy(), B_min, P)
    print(shape, theta, B_min, s)


@pytest.mark.parametrize("mode", ["dense", "mask", "lists"])
def test_standalone_decode_modes(eti, mode):
    """eti_paged_decode without precomputed scores: dense, from a mask, from lists."""
    w = workloads.Workload("d", B=4, Hq=32, Hkv=8, D=128, P=16, V=16, ctx=("list", [50, 700, 1, 333]),
                           seed=8, hi_frac=0.05)
    kv = workloads.make_kv(w, DEV, poison_tail=True)
    n = parity.host_kv(kv)
    rng = np.random.default_rng(1)
    mask = (rng.random((w.B, w.Hkv, w.max_blocks)) < 0.6).astype(np.uint8)
    for b, L in enumerate(n["L"]):
        mask[b, :, -(-int(L) // w.P):] = 0
    out = torch.empty((w.B, w.Hq, w.D), dtype=torch.bfloat16, device=DEV)
    err = torch.empty(w.B, dtype=torch.int32, device=DEV)
    ws = torch.empty(eti.paged_decode_workspace_size(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, False),
                     dtype=torch.uint8, device=DEV)
    kw = {}
    if mode == "mask":
        kw["keep_mask"] = torch.from_numpy(mask).to(DEV)
    elif mode == "lists":
        idx = np.full(mask.shape, -1, np.int32)
        cnt = mask.sum(-1).astype(np.int32)
        for b in range(w.B):
            for h in range(w.Hkv):
                nz = np.nonzero(mask[b, h])[0][::-1]   # any order is accepted
                idx[b, h, :len(nz)] = nz
        kw["kept_idx"] = torch.from_numpy(idx).to(DEV)
        kw["kept_cnt"] = torch.from_numpy(cnt).to(DEV)
    eti.eti_paged_decode(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                         kv["scale"], out, err, ws, **kw)
    torch.cuda.synchronize()
    ref, rerr = oracle.paged_attention(n["q"], n["k"], n["v"], n["bt"], n["L"], n["scale"],
                                       None if mode == "dense" else mask)
    parity.compare_attention(out.float().cpu().numpy(), ref)
    assert np.array_equal(err.cpu().numpy().view(np.uint32), rerr)


def test_attention_maximum_batch(eti):
    """The largest batch the attention calls accept (8192 sequences): the
    scorer's per-sequence prefix no longer leaves room for two CTAs per SM.
    Ragged contexts of 0 to 100 tokens (empty sequences included), every
    sequence against the oracle."""
    B = 8192
    lens = np.random.default_rng(9).integers(0, 101, B)
    lens[::97] = 0
    w = workloads.Workload("mb", B=B, Hq=8, Hkv=2, D=64, P=16, V=16, ctx=("list", [int(x) for x in lens]),
                           seed=9, hi_frac=0.05)
    kv = workloads.make_kv(w, DEV)
    th = torch.full((B,), 0.9, dtype=torch.float32, device=DEV)
    st = _step(eti, w, kv, th, 2)
    s = _check_step(st, parity.host_kv(kv), th.cpu().numpy(), 2, w.P)
    print(s)


@pytest.mark.parametrize("mode", ["dense", "mask", "lists"])
def test_standalone_decode_long_segments(eti, mode):
    """eti_paged_decode without precomputed scores on segments of up to 8192
    blocks: its internal keep-set pass takes the wide kernel on a pair of CTAs
    per segment; dense, from a mask, from lists."""
    w = workloads.Workload("dl", B=2, Hq=32, Hkv=8, D=128, P=16, V=16, ctx=("list", [40000, 131072]),
                           seed=17, hi_frac=0.02)
    kv = workloads.make_kv(w, DEV)
    n = parity.host_kv(kv)
    rng = np.random.default_rng(3)
    mask = (rng.random((w.B, w.Hkv, w.max_blocks)) < 0.3).astype(np.uint8)
    for b, L in enumerate(n["L"]):
        mask[b, :, -(-int(L) // w.P):] = 0
    out = torch.empty((w.B, w.Hq, w.D), dtype=torch.bfloat16, device=DEV)
    err = torch.empty(w.B, dtype=torch.int32, device=DEV)
    ws = torch.empty(eti.paged_decode_workspace_size(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, False),
                     dtype=torch.uint8, device=DEV)
    kw = {}
    if mode == "mask":
        kw["keep_mask"] = torch.from_numpy(mask).to(DEV)
    elif mode == "lists":
        idx = np.full(mask.shape, -1, np.int32)
        cnt = mask.sum(-1).astype(np.int32)
        for b in range(w.B):
            for h in range(w.Hkv):
                nz = np.nonzero(mask[b, h])[0]
                rng.shuffle(nz)                       # any order is accepted
                idx[b, h, :len(nz)] = nz
        kw["kept_idx"] = torch.from_numpy(idx).to(DEV)
        kw["kept_cnt"] = torch.from_numpy(cnt).to(DEV)
    eti.eti_paged_decode(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                         kv["scale"], out, err, ws, num_pages=kv["num_pages"], **kw)
    torch.cuda.synchronize()
    ref, rerr = oracle.paged_attention(n["q"], n["k"], n["v"], n["bt"], n["L"], n["scale"],
                                       None if mode == "dense" else mask, num_pages=n["num_pages"])
    print(mode, parity.compare_attention(out.float().cpu().numpy(), ref))
    assert np.array_equal(err.cpu().numpy().view(np.uint32), rerr)


def test_attention_edge_cases(eti):
    """Empty sequences, a bad page id and a bad context length: error bits and zero outputs."""
    w = workloads.Workload("e", B=4, Hq=8, Hkv=2, D=64, P=16, V=16, ctx=("list", [0, 40, 40, 40]),
                           seed=31)
    kv = workloads.make_kv(w, DEV)
    kv["block_table"][2, 1] = kv["num_pages"] + 7
    kv["ctx_lens"][3] = w.max_blocks * w.P + 5
    th = torch.zeros(w.B, device=DEV)
    st = _step(eti, w, kv, th, 1)
    n = parity.host_kv(kv)
    ref = oracle.score_prune(n["q"], n["k"], n["bt"], n["L"], n["scale"], th.cpu().numpy(), 1)
    assert list(ref["err"]) == [0, 0, 1, 2]
    assert np.array_equal(st.err_attn.cpu().numpy().view(np.uint32), ref["err"])
    assert np.array_equal(st.err_dec.cpu().numpy().view(np.uint32), ref["err"])
    out = st.out.float().cpu().numpy()
    assert (out[[0, 2, 3]] == 0).all() and np.abs(out[1]).sum() > 0
    assert (st.kept_cnt.cpu().numpy()[[0, 2, 3]] == 0).all()


def test_page_permutation_and_repeat_invariance(eti):
    w = workloads.Workload("perm", B=3, Hq=16, Hkv=4, D=128, P=16, V=16, ctx=("list", [300, 45, 1000]),
                           seed=41, hi_frac=0.1)
    kv = workloads.make_kv(w, DEV)
    th = torch.full((w.B,), 0.9, device=DEV)
    a = _step(eti, w, kv, th, 2)
    out_a, mask_a = a.out.clone(), a.keep_mask.clone()
    perm = torch.randperm(kv["num_pages"], generator=torch.Generator().manual_seed(0)).to(DEV)
    inv = torch.empty_like(perm)
    inv[perm] = torch.arange(len(perm), device=DEV)
    kv2 = dict(kv, k_cache=kv["k_cache"][perm].contiguous(), v_cache=kv["v_cache"][perm].contiguous(),
               block_table=torch.where(kv["block_table"] >= 0,
                                       inv[kv["block_table"].clamp(min=0).long()].int(),
                                       kv["block_table"]))
    b = _step(eti, w, kv2, th, 2)
    assert torch.equal(mask_a, b.keep_mask)
    assert torch.equal(out_a, b.out)
    c = _step(eti, w, kv, th, 2)
    assert torch.equal(out_a, c.out)


# ---------------------------------------------------------------------------
# full-size workloads (benchmark launch configuration), sampled oracle checks

def _pool_for(w):
    if w.pool is None:
        return None
    free, _ = torch.cuda.mem_get_info()
    page_bytes = 2 * w.Hkv * w.P * w.D * 2
    cap = int(0.25 * free // page_bytes)
    return min(w.pool, 1 << max(10, cap.bit_length() - 1))


@pytest.mark.parametrize("name,nsample", [("tiny", 4), ("llama3_8b", 64), ("long_ctx", 8),
                                          ("mixed_batch", 256), ("llama3_70b", 16)])
def test_attention_full_workloads(eti, name, nsample):
    """The step at full size in the benchmark's launch configuration: every
    sequence of tiny, llama3_8b, long_ctx and mixed_batch and 16 of the 128
    llama3_70b sequences (scores, keep set, kept lists, output, error words)
    against the oracle on their gathered pages."""
    w = workloads.WORKLOADS[name]
    kv = workloads.make_kv(w, DEV, pool=_pool_for(w))
    lg = workloads.make_logits(w, DEV)
    g = parity.run_ets(eti, lg, seed=w.seed)          # theta from this step's entropy
    theta = torch.from_numpy(g["theta_next"]).to(DEV)
    B_min = 1
    st = _step(eti, w, kv, theta, B_min)
    rng = np.random.default_rng(w.seed)
    seqs = sorted(rng.choice(w.B, size=min(nsample, w.B), replace=False).tolist())
    sub = parity.host_from_gather(workloads.gather_sequences(kv, seqs))
    s = _check_step(st, sub, theta.cpu().numpy()[seqs], B_min, w.P, seqs=seqs)
    assert len(seqs) == min(nsample, w.B)
    kept = st.kept_cnt.sum().item()
    total = sum(-(-int(L) // w.P) for L in kv["ctx_lens"].cpu().numpy()) * w.Hkv
    print(name, s, f"kept fraction {kept / total:.3f}")
    assert torch.isfinite(st.out.float()).all()


def test_long_context_keep_fraction_sweep(eti):
    """The long-context sweep: theta = +inf and B_min = ceil(f n_b), f = 0.1..1.0."""
    w = workloads.WORKLOADS["long_ctx"].scaled(B=3)
    kv = workloads.make_kv(w, DEV)
    th = torch.full((w.B,), float("inf"), device=DEV)
    seqs = [0, 2]
    sub = parity.host_from_gather(workloads.gather_sequences(kv, seqs))
    L = kv["ctx_lens"].cpu().numpy()
    for f in (0.1, 0.5, 1.0):
        # one B_min for the batch: the fraction of the longest sequence
        B_min = int(math.ceil(f * -(-int(L.max()) // w.P)))
        st = _step(eti, w, kv, th, B_min)
        cnt = st.kept_cnt.cpu().numpy()
        nb = -(-L // w.P)
        assert (cnt == np.minimum(B_min, nb)[:, None]).all()
        _check_step(st, sub, th.cpu().numpy()[seqs], B_min, w.P, seqs=seqs)
