"""A sequence's results do not depend on the batch around it.

The scorer splits the flattened (sequence, kv head, block) list evenly over
its warps, and the decode splits the kept blocks of all segments over its
warps (split segments are merged in warp order), so a sequence decoded alone
is split differently from the same sequence inside a batch.  Its block
scores and keep set are computed per block and per segment and must be
identical bit for bit; its attention output is the same sum taken over
other split points, so it may differ only by the rounding of the
re-associated fp32 sums and of the bf16 store.
"""
import numpy as np
import pytest
import torch

import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _attend(eti, w, B, q, bt, L, kv, theta):
    st = eti.DecodeStep(B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, w.V, device=DEV)
    st.attention(q, kv["k_cache"], kv["v_cache"], bt, L, kv["scale"], theta, 2,
                 num_pages=kv["num_pages"])
    torch.cuda.synchronize()
    return st


def test_sequence_alone_equals_sequence_in_batch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2603_03310_gb300 as eti
    eti.build()
    eti.load()
    w = workloads.Workload("split", B=6, Hq=32, Hkv=8, D=128, P=16, V=16,
                           ctx=("list", [5000, 17, 2048, 900, 8000, 64]), seed=61, hi_frac=0.05)
    kv = workloads.make_kv(w, DEV)
    theta = torch.full((w.B,), 0.5, dtype=torch.float32, device=DEV)
    full = _attend(eti, w, w.B, kv["q"], kv["block_table"], kv["ctx_lens"], kv, theta)
    for b in range(w.B):
        one = _attend(eti, w, 1, kv["q"][b:b + 1], kv["block_table"][b:b + 1],
                      kv["ctx_lens"][b:b + 1], kv, theta[b:b + 1])
        for name in ("keep_mask", "kept_idx", "kept_cnt", "block_score", "kept_norm", "err_attn",
                     "err_dec"):
            assert torch.equal(getattr(full, name)[b], getattr(one, name)[0]), (b, name)
        a = full.out[b].float().cpu().numpy()
        c = one.out[0].float().cpu().numpy()
        # two bf16 ulps of the larger value (the fp32 sums differ in the last bits)
        tol = 2.0 ** -7 * np.maximum(np.abs(a), np.abs(c)) + 1e-3
        assert np.all(np.abs(a - c) <= tol), (b, float(np.max(np.abs(a - c))))
