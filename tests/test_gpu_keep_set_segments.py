"""The keep set on the Llama-3-70B head shape: g = 8 query heads per kv head
and segments of up to 2048 blocks, the shape the segment kernel serves (the
terms of a segment in shared memory, one CTA per segment, the budget and the
compaction per block).  Against the oracle through the C ABI: block scores
(2e-5 plus the fp32 band), keep masks, kept lists and counts (exact except
counted near-ties), error words, the kept-token normaliser through the
pruned decode's output, for thresholds, budgets (the argmax and the radix
select, ties to the lower index) and the three score modes.
"""
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


@pytest.fixture(scope="module")
def case():
    # one full-length segment, a short one, a ragged last block, an empty sequence
    w = workloads.Workload("seg", B=4, Hq=64, Hkv=8, D=128, P=16, V=16,
                           ctx=("list", [32768, 1000, 17001, 0]), seed=77, hi_frac=0.05)
    kv = workloads.make_kv(w, DEV, poison_tail=True)
    return w, kv, parity.host_kv(kv)


def _store(kv, seed):
    pages, _, P, _ = kv["k_cache"].shape
    g = torch.Generator().manual_seed(seed)
    return torch.empty(pages, P).exponential_(0.5, generator=g).to(DEV)


@pytest.mark.parametrize("theta,B_min", [(0.0, 1), (0.9, 1), (float("inf"), 1), (1.2, 0),
                                         (float("inf"), 700), (0.7, 300), (0.5, 10 ** 6)])
def test_segment_keep_set_and_decode(eti, case, theta, B_min):
    w, kv, n = case
    th = torch.full((w.B,), theta, dtype=torch.float32, device=DEV)
    st = eti.DecodeStep(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, w.V, device=DEV)
    st.attention(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"], kv["scale"],
                 th, B_min, num_pages=kv["num_pages"])
    torch.cuda.synchronize()
    th_np = th.cpu().numpy()
    ref = oracle.score_prune(n["q"], n["k"], n["bt"], n["L"], n["scale"], th_np, B_min,
                             num_pages=n["num_pages"], want_heads=True)
    band = parity.score_bands(ref, n)
    gm = st.keep_mask.cpu().numpy()
    worst = parity.compare_scores(st.block_score.cpu().numpy(), ref["block_score"], w.P, n["L"], band)
    ties = parity.compare_masks(gm, st.kept_idx.cpu().numpy(), st.kept_cnt.cpu().numpy(), ref, th_np,
                                B_min, w.P, n["L"], band)
    assert np.array_equal(st.err_attn.cpu().numpy().view(np.uint32), ref["err"])
    if np.isinf(theta) and 0 < B_min < 10 ** 6:
        nb = -(-n["L"] // w.P)
        assert (st.kept_cnt.cpu().numpy() == np.minimum(B_min, nb)[:, None]).all()
    out_ref, err = oracle.paged_attention(n["q"], n["k"], n["v"], n["bt"], n["L"], n["scale"], gm,
                                          num_pages=n["num_pages"])
    out_err = parity.compare_attention(st.out.float().cpu().numpy(), out_ref)
    assert np.array_equal(st.err_dec.cpu().numpy().view(np.uint32), err)
    print(theta, B_min, dict(score_err=worst, out_err=out_err, **ties))


@pytest.mark.parametrize("mode", [1, 2])
@pytest.mark.parametrize("theta,B_min", [(0.9, 1), (float("inf"), 700)])
def test_segment_score_modes(eti, case, mode, theta, B_min):
    w, kv, n = case
    store = _store(kv, 5)
    f32, i32, u8 = torch.float32, torch.int32, torch.uint8
    shp = (w.B, w.Hkv, w.max_blocks)
    out = dict(keep_mask=torch.empty(shp, dtype=u8, device=DEV),
               kept_idx=torch.empty(shp, dtype=i32, device=DEV),
               kept_cnt=torch.empty((w.B, w.Hkv), dtype=i32, device=DEV),
               block_score=torch.empty(shp, dtype=f32, device=DEV),
               err=torch.empty(w.B, dtype=i32, device=DEV))
    ws = torch.empty(eti.score_prune_workspace_size(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks),
                     dtype=u8, device=DEV)
    th = torch.full((w.B,), theta, dtype=torch.float32, device=DEV)
    eti.eti_score_prune_blocks(kv["q"], kv["k_cache"], kv["block_table"], kv["ctx_lens"], kv["scale"],
                               th, B_min, out["keep_mask"], out["kept_idx"], out["kept_cnt"], out["err"],
                               ws, block_score=out["block_score"], num_pages=kv["num_pages"],
                               score_mode=mode, tok_surp=store if mode == 1 else None)
    torch.cuda.synchronize()
    got = {k: v.cpu().numpy() for k, v in out.items()}
    th_np = th.cpu().numpy()
    ref = oracle.score_prune(n["q"], n["k"], n["bt"], n["L"], n["scale"], th_np, B_min,
                             num_pages=n["num_pages"], want_heads=True, score_mode=mode,
                             surp=store.cpu().numpy())
    band = parity.score_bands(ref, n, score_mode=mode)
    parity.compare_scores(got["block_score"], ref["block_score"], w.P, n["L"], band)
    parity.compare_masks(got["keep_mask"], got["kept_idx"], got["kept_cnt"], ref, th_np, B_min, w.P,
                         n["L"], band)
    assert np.array_equal(got["err"].view(np.uint32), ref["err"])
