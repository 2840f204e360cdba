"""The seeded synthetic inputs follow their stated recipe (CPU only).

Both sides of every parity check read these tensors, so a generator that
drifted from the recipe (shared pages, lengths out of range, a missing spike)
would weaken every test without failing any.  These checks pin the recipe:
context-length ranges, page tables drawn from a permutation of the pool,
-1 past each sequence's last block, the high-norm key chunks, the logit
spikes, the controller state, determinism per seed, and the host gather used
for spot checks of large workloads.
"""
import math

import numpy as np
import pytest
import torch

import workloads
from workloads import WORKLOADS


@pytest.mark.parametrize("name", sorted(WORKLOADS))
def test_context_lengths_follow_the_recipe(name):
    w = WORKLOADS[name]
    L = workloads.ctx_lengths(w)
    assert L.dtype == np.int32 and L.shape == (w.B,)
    if w.ctx[0] == "list":
        assert L.tolist() == list(w.ctx[1])
    else:
        assert L.min() >= w.ctx[1] and L.max() <= w.ctx[2]
        assert w.max_blocks == -(-w.ctx[2] // w.P)
        assert len(np.unique(L)) > w.B // 2          # drawn, not constant
    if w.ctx[0] == "loguniform":
        # log-uniform: the median sits near the geometric mean of the range
        gm = math.sqrt(w.ctx[1] * w.ctx[2])
        assert gm / 3 < np.median(L) < gm * 3
    assert np.array_equal(L, workloads.ctx_lengths(w))  # seeded


def _small(name, **kw):
    w = WORKLOADS[name]
    return w.scaled(**{**dict(B=12, ctx=("uniform", 1, 40 * w.P)), **kw})


@pytest.mark.parametrize("pool", [None, 5000])
def test_block_tables_use_distinct_pages_from_the_pool(pool):
    w = _small("llama3_8b", hi_frac=0.25)
    kv = workloads.make_kv(w, "cpu", pool=pool)
    bt, L = kv["block_table"].numpy(), kv["ctx_lens"].numpy()
    nb = (L + w.P - 1) // w.P
    used = np.concatenate([bt[b, :nb[b]] for b in range(w.B)])
    assert len(np.unique(used)) == len(used) == nb.sum()   # no page shared
    assert used.min() >= 0 and used.max() < kv["num_pages"]
    assert kv["num_pages"] == (pool or nb.sum())
    for b in range(w.B):
        assert (bt[b, nb[b]:] == -1).all()
    if pool:
        # a permutation of the whole pool: the used ids are spread over it
        assert used.max() > pool // 2
    assert kv["k_cache"].shape == (kv["num_pages"], w.Hkv, w.P, w.D)
    assert kv["k_cache"].dtype == kv["v_cache"].dtype == kv["q"].dtype == torch.bfloat16
    assert kv["scale"] == pytest.approx(1 / math.sqrt(w.D))


def test_high_norm_key_chunks_are_scaled_by_four():
    w = _small("llama3_8b", hi_frac=0.3, B=16)
    kv = workloads.make_kv(w, "cpu")
    hi, ids = kv["hi_chunks"], kv["page_ids"]
    assert 0.15 < hi.mean() < 0.45
    kn = kv["k_cache"].float()[torch.from_numpy(ids)].pow(2).mean(dim=(2, 3)).sqrt().numpy()
    vn = kv["v_cache"].float()[torch.from_numpy(ids)].pow(2).mean(dim=(2, 3)).sqrt().numpy()
    # rms of P*D standard normals is ~1; high-norm chunks ~4; V is never scaled
    assert np.all(np.abs(kn[hi] - 4.0) < 0.6) and np.all(np.abs(kn[~hi] - 1.0) < 0.15)
    assert np.all(np.abs(vn - 1.0) < 0.15)


def test_logits_and_controller_state_follow_the_recipe():
    w = WORKLOADS["llama3_8b"].scaled(B=40, V=20000)
    lg = workloads.make_logits(w, "cpu")
    z = lg["logits"].numpy().astype(np.float64)
    logV = math.log(w.V)
    # per-row scale s_b log-uniform on [0.1, 10]: the robust spread of each row
    s = (np.quantile(z, 0.75, axis=1) - np.quantile(z, 0.25, axis=1)) / 1.349
    assert s.min() > 0.08 and s.max() < 11 and s.min() < 0.5 and s.max() > 2
    H_prev = lg["H_prev"].numpy()
    assert H_prev.min() >= 0 and H_prev.max() <= logV
    assert np.allclose(lg["H_target"].numpy(), 0.5 * logV, rtol=1e-6)
    assert (lg["T_in"].numpy() == 1).all() and (lg["tau"].numpy() == 0).all()
    # seeded
    again = workloads.make_logits(w, "cpu")
    assert torch.equal(again["logits"], lg["logits"]) and torch.equal(again["H_prev"], lg["H_prev"])


def _spikes(w):
    """Per row, the offsets added on top of the s_b * N(0, 1) bulk: the same
    workload with zero spikes draws the same bulk (its own generator)."""
    z = workloads.make_logits(w, "cpu")["logits"].numpy().astype(np.float64)
    bulk = workloads.make_logits(w.scaled(spike=0.0, even_row_spike=None), "cpu")["logits"]
    d = z - bulk.numpy().astype(np.float64)
    return [d[b][np.abs(d[b]) > 1e-3] for b in range(w.B)], [np.nonzero(np.abs(d[b]) > 1e-3)[0]
                                                             for b in range(w.B)]


def test_spiked_tokens_follow_the_recipe():
    # 0-3 distinct tokens per row at +8, the count uniform on {0, 1, 2, 3}
    w = WORKLOADS["llama3_8b"].scaled(B=200, V=3000)
    add, where = _spikes(w)
    counts = [len(a) for a in add]
    assert set(counts) == {0, 1, 2, 3}
    assert all(np.allclose(a, 8.0, atol=1e-4) for a in add)
    assert all(len(set(x.tolist())) == len(x) for x in where)
    assert 0.15 < counts.count(0) / len(counts) < 0.35
    # mixed batch: every even row one token at +20, odd rows the 0-3 at +8
    w = WORKLOADS["mixed_batch"].scaled(B=40, V=3000)
    add, _ = _spikes(w)
    for b, a in enumerate(add):
        if b % 2 == 0:
            assert len(a) == 1 and abs(a[0] - 20.0) < 1e-4
        else:
            assert len(a) <= 3 and np.allclose(a, 8.0, atol=1e-4)


def test_strided_logits_pad_with_nan_past_V():
    w = WORKLOADS["tiny"]
    lg = workloads.make_logits(w, "cpu", ld=w.V + 13)
    z = lg["logits"].numpy()
    assert z.shape == (w.B, w.V + 13) and lg["ld"] == w.V + 13
    assert np.isnan(z[:, w.V:]).all() and np.isfinite(z[:, :w.V]).all()
    plain = workloads.make_logits(w, "cpu")["logits"].numpy()
    assert np.array_equal(z[:, :w.V], plain)


def test_poisoned_tail_slots_only_past_each_sequence_end():
    w = WORKLOADS["tiny"].scaled(ctx=("list", [5, 16, 33, 0]))
    kv = workloads.make_kv(w, "cpu", poison_tail=True)
    bt, L = kv["block_table"].numpy(), kv["ctx_lens"].numpy()
    k = kv["k_cache"].float().numpy()
    for b in range(w.B):
        nb = -(-int(L[b]) // w.P)
        for j in range(nb):
            page = k[bt[b, j]]
            valid = min(w.P, int(L[b]) - j * w.P)
            assert np.isfinite(page[:, :valid]).all()
            assert np.isnan(page[:, valid:]).all()


def test_gather_sequences_is_a_compact_copy_of_their_pages():
    w = _small("llama3_8b", B=6)
    kv = workloads.make_kv(w, "cpu", pool=900)
    seqs = [4, 1]
    sub = workloads.gather_sequences(kv, seqs)
    P = w.P
    kbits, vbits = workloads.bf16_bits(kv["k_cache"]), workloads.bf16_bits(kv["v_cache"])
    for i, b in enumerate(seqs):
        L = int(kv["ctx_lens"][b])
        assert sub["ctx_lens"][i] == L
        for j in range(-(-L // P)):
            src = int(kv["block_table"][b, j])
            dst = sub["block_table"][i, j]
            assert np.array_equal(sub["k_cache"][dst], kbits[src])
            assert np.array_equal(sub["v_cache"][dst], vbits[src])
    assert np.array_equal(sub["q"], workloads.bf16_bits(kv["q"][seqs]))
    assert sub["num_pages"] == len(sub["pages"])
