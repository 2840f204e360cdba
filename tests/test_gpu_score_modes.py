"""Score modes of the block score (Section 3.2) and the fused surprisal store.

Mode E reads I(v_i) as the stored surprisal of token i (a paged store
[num_pages][P] written by the sampling call), mode M as 1 (the block's
attention mass).  Both go through the C ABI against the oracle on the same
seeded inputs: block scores within 2e-5 plus the fp32 evaluation band (4 |dx|
in these modes), keep sets exact except for counted near-ties.  The sampling
call's surp_store output must hold exactly the tok_surprisal it returns, at
the given slots and nowhere else.
"""
import numpy as np
import pytest
import torch

import oracle
import parity
import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
MODES = [(1, "E"), (2, "M")]


@pytest.fixture(scope="module")
def eti():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as m
    m.build()
    m.load()
    oracle.build()
    return m


def _store(kv, seed):
    """A surprisal store shaped like the key pages, values ~ Exp(mean 2) (seeded)."""
    pages, _, P, _ = kv["k_cache"].shape
    g = torch.Generator().manual_seed(seed)
    return torch.empty(pages, P).exponential_(0.5, generator=g).to(DEV)


def _score_prune(eti, w, kv, theta, B_min, mode, store):
    f32, i32, u8 = torch.float32, torch.int32, torch.uint8
    shp = (w.B, w.Hkv, w.max_blocks)
    out = dict(keep_mask=torch.empty(shp, dtype=u8, device=DEV),
               kept_idx=torch.empty(shp, dtype=i32, device=DEV),
               kept_cnt=torch.empty((w.B, w.Hkv), dtype=i32, device=DEV),
               block_score=torch.empty(shp, dtype=f32, device=DEV),
               err=torch.empty(w.B, dtype=i32, device=DEV))
    ws = torch.empty(eti.score_prune_workspace_size(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks),
                     dtype=u8, device=DEV)
    eti.eti_score_prune_blocks(kv["q"], kv["k_cache"], kv["block_table"], kv["ctx_lens"], kv["scale"],
                               theta, B_min, out["keep_mask"], out["kept_idx"], out["kept_cnt"],
                               out["err"], ws, block_score=out["block_score"],
                               num_pages=kv["num_pages"], score_mode=mode,
                               tok_surp=store if mode == 1 else None)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _check(got, n, store_np, theta_np, B_min, mode, seqs=None):
    rng = slice(None) if seqs is None else seqs
    ref = oracle.score_prune(n["q"], n["k"], n["bt"], n["L"], n["scale"], theta_np, B_min,
                             num_pages=n.get("num_pages"), want_heads=True, score_mode=mode,
                             surp=store_np)
    band = parity.score_bands(ref, n, score_mode=mode)
    P = n["k"].shape[2]
    worst = parity.compare_scores(got["block_score"][rng], ref["block_score"], P, n["L"], band)
    ties = parity.compare_masks(got["keep_mask"][rng], got["kept_idx"][rng], got["kept_cnt"][rng],
                                ref, theta_np, B_min, P, n["L"], band)
    assert np.array_equal(got["err"][rng].view(np.uint32), ref["err"])
    return dict(score_err=worst, **ties)


SHAPES = [
    # (B, Hq, Hkv, D, P, lens)
    (4, 8, 8, 64, 16, [64, 128, 192, 256]),
    (3, 32, 8, 128, 16, [1, 37, 1000]),
    (5, 16, 2, 128, 32, [33, 64, 500, 17, 2049]),
    (2, 24, 3, 128, 32, [800, 95]),
]


@pytest.mark.parametrize("mode,name", MODES)
@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("theta,B_min", [(0.8, 1), (1.0, 3), (float("inf"), 2)])
def test_score_modes_small(eti, mode, name, shape, theta, B_min):
    B, Hq, Hkv, D, P, lens = shape
    w = workloads.Workload("m", B=B, Hq=Hq, Hkv=Hkv, D=D, P=P, V=16, ctx=("list", lens),
                           seed=sum(lens) + D + P + mode, hi_frac=0.1)
    kv = workloads.make_kv(w, DEV, poison_tail=True)
    store = _store(kv, seed=B + mode)
    th = torch.full((B,), theta, dtype=torch.float32, device=DEV)
    got = _score_prune(eti, w, kv, th, B_min, mode, store)
    s = _check(got, parity.host_kv(kv), store.cpu().numpy(), th.cpu().numpy(), B_min, mode)
    print(name, shape, theta, B_min, s)


@pytest.mark.parametrize("mode,name", MODES)
def test_score_modes_llama3_8b(eti, mode, name):
    """Full-size step (64 sequences, contexts up to 8192), sampled sequences
    checked against the oracle through gathered pages and store rows."""
    w = workloads.WORKLOADS["llama3_8b"]
    kv = workloads.make_kv(w, DEV)
    store = _store(kv, seed=77 + mode)
    th = torch.full((w.B,), 0.9, dtype=torch.float32, device=DEV)
    got = _score_prune(eti, w, kv, th, 1, mode, store)
    seqs = [3, 17, 40, 63]
    sub = parity.host_from_gather(workloads.gather_sequences(kv, seqs))
    store_sub = store.cpu().numpy()[sub["pages"]]
    s = _check(got, sub, store_sub, th.cpu().numpy()[seqs], 1, mode, seqs=seqs)
    kept = got["kept_cnt"].sum() / sum(-(-int(L) // w.P) * w.Hkv for L in kv["ctx_lens"].cpu().numpy())
    print(name, s, f"kept fraction {kept:.3f}")


@pytest.mark.parametrize("mode", [0, 1, 2])
def test_two_calls_equal_fused_call(eti, mode):
    """eti_score_blocks (with the store) + eti_prune_blocks (with the mode)
    gives the fused call's keep set and scores bit for bit."""
    w = workloads.Workload("t", B=3, Hq=32, Hkv=8, D=128, P=16, V=16, ctx=("list", [900, 33, 2000]),
                           seed=4, hi_frac=0.05)
    kv = workloads.make_kv(w, DEV)
    store = _store(kv, seed=5)
    th = torch.full((w.B,), 1.0, dtype=torch.float32, device=DEV)
    fused = _score_prune(eti, w, kv, th, 2, mode, store)
    g = w.Hq // w.Hkv
    stats = torch.empty((w.B, w.Hkv, w.max_blocks, g, 4), dtype=torch.float32, device=DEV)
    eti.eti_score_blocks(kv["q"], kv["k_cache"], kv["block_table"], kv["ctx_lens"], kv["scale"],
                         stats, num_pages=kv["num_pages"], tok_surp=store if mode == 1 else None)
    shp = (w.B, w.Hkv, w.max_blocks)
    km = torch.empty(shp, dtype=torch.uint8, device=DEV)
    ki = torch.empty(shp, dtype=torch.int32, device=DEV)
    kc = torch.empty((w.B, w.Hkv), dtype=torch.int32, device=DEV)
    bs = torch.empty(shp, dtype=torch.float32, device=DEV)
    err = torch.empty(w.B, dtype=torch.int32, device=DEV)
    eti.eti_prune_blocks(stats, kv["block_table"], kv["ctx_lens"], (w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks),
                         th, 2, km, ki, kc, err, block_score=bs, num_pages=kv["num_pages"], score_mode=mode)
    torch.cuda.synchronize()
    assert np.array_equal(km.cpu().numpy(), fused["keep_mask"])
    assert np.array_equal(kc.cpu().numpy(), fused["kept_cnt"])
    assert np.array_equal(bs.cpu().numpy(), fused["block_score"])


@pytest.mark.parametrize("noalloc", [False, True])
def test_fused_surprisal_store(eti, noalloc):
    """store[slot[b]] = tok_surprisal[b] exactly, for rows without an error bit
    and slots inside [0, num_slots); every other entry keeps its value."""
    w = workloads.WORKLOADS["llama3_8b"].scaled(B=24)
    lg = workloads.make_logits(w, DEV)
    lg["logits"][5, 100] = float("nan")          # an error row: nothing is stored for it
    B = w.B
    n_slots = 4096
    store = torch.full((n_slots,), -5.0, dtype=torch.float32, device=DEV)
    rng = np.random.default_rng(2)
    slots = rng.choice(n_slots, size=B, replace=False).astype(np.int64)
    slots[7] = -1                                # skipped
    slots[11] = n_slots + 3                      # outside the store: skipped
    slot_t = torch.from_numpy(slots).to(DEV)
    f32, i32 = torch.float32, torch.int32
    o = {k: torch.empty(B, dtype=f32, device=DEV) for k in ("H", "T_out", "surp")}
    tok = torch.empty(B, dtype=i32, device=DEV)
    err = torch.empty(B, dtype=i32, device=DEV)
    tau = lg["tau"].clone()
    args = (lg["logits"], lg["T_in"], lg["H_prev"], tau, lg["H_target"], tok, o["H"], o["T_out"], err)
    kw = dict(seed=3, offset=1, tok_surprisal=o["surp"], surp_store=store, slot_mapping=slot_t)
    if noalloc:
        eti.eti_entropy_temp_sample_noalloc(*args, **kw)
    else:
        ws = torch.empty(eti.entropy_temp_sample_workspace_size(B, w.V), dtype=torch.uint8, device=DEV)
        eti.eti_entropy_temp_sample(*args, ws, **kw)
    torch.cuda.synchronize()
    st, sp, e = store.cpu().numpy(), o["surp"].cpu().numpy(), err.cpu().numpy()
    assert e[5] != 0 and (np.delete(e, 5) == 0).all()
    written = np.zeros(n_slots, bool)
    for b in range(B):
        if e[b] == 0 and 0 <= slots[b] < n_slots:
            assert st[slots[b]] == sp[b], b          # the same fp32 value, bit for bit
            written[slots[b]] = True
    assert (st[~written] == -5.0).all()
    assert written.sum() == B - 3
    # the stored values are what the oracle gives for the drawn tokens
    r = parity.oracle_ets(lg, seed=3, offset=1)
    ok = (e == 0) & (r["tok"] == tok.cpu().numpy())
    assert np.allclose(sp[ok], r["surprisal"][ok], rtol=1e-4, atol=1e-5)


@pytest.mark.parametrize("mode,name", [(0, "A")] + MODES)
def test_score_modes_long_segments(eti, mode, name):
    """Segments past the register-resident layout (up to 8192 blocks with
    g = 4): the keep set comes from the wide kernel with its shared-memory
    cache of the block terms, in all three score modes."""
    w = workloads.Workload("wl", B=2, Hq=32, Hkv=8, D=128, P=16, V=16, ctx=("list", [40000, 131072]),
                           seed=21 + mode, hi_frac=0.02)
    kv = workloads.make_kv(w, DEV)
    store = _store(kv, seed=3 + mode)
    th = torch.full((w.B,), 0.9, dtype=torch.float32, device=DEV)
    got = _score_prune(eti, w, kv, th, 3, mode, store)
    s = _check(got, parity.host_kv(kv), store.cpu().numpy(), th.cpu().numpy(), 3, mode)
    print(name, s)


def test_prune_long_segment_without_term_cache(eti):
    """12,500 blocks with g = 4 need more than the 200 KB term cache: the wide
    kernel recomputes the terms from the stats; a budget select as well."""
    w = workloads.Workload("wn", B=1, Hq=32, Hkv=8, D=128, P=16, V=16, ctx=("list", [200000]),
                           seed=31, hi_frac=0.02)
    assert w.max_blocks * 4 * (1 + 4) > 200 * 1024
    kv = workloads.make_kv(w, DEV)
    th = torch.full((w.B,), 1.2, dtype=torch.float32, device=DEV)
    got = _score_prune(eti, w, kv, th, 700, 0, None)
    s = _check(got, parity.host_kv(kv), None, th.cpu().numpy(), 700, 0)
    print(s)


@pytest.mark.parametrize("B_min", [3000, 5000])
def test_budget_ties_across_a_cluster(eti, B_min):
    """q = 0 gives every full block the same stats, hence bitwise-equal group
    scores: with theta = +inf the kept blocks of every head are exactly blocks
    0..B_min-1, whichever CTA of the pair holds them (8192 blocks: the
    segment is split between two CTAs at block 4096, so B_min = 5000 takes
    all of the first CTA's blocks and the first 904 of the second's)."""
    w = workloads.Workload("tie", B=1, Hq=32, Hkv=8, D=128, P=16, V=16, ctx=("list", [131072]), seed=41,
                           hi_frac=0.0)
    kv = workloads.make_kv(w, DEV)
    kv["q"].zero_()
    th = torch.full((w.B,), float("inf"), dtype=torch.float32, device=DEV)
    got = _score_prune(eti, w, kv, th, B_min, 0, None)
    want = np.zeros((w.B, w.Hkv, w.max_blocks), np.uint8)
    want[:, :, :B_min] = 1
    assert np.array_equal(got["keep_mask"], want)
    assert (got["kept_cnt"] == B_min).all()
    assert np.array_equal(got["kept_idx"][:, :, :B_min], np.broadcast_to(np.arange(B_min), (w.B, w.Hkv, B_min)))
    assert (got["kept_idx"][:, :, B_min:] == -1).all()
    sc = got["block_score"][0, :, :8192]
    assert (sc == sc[:, :1]).all()                  # every block the same score, bit for bit
