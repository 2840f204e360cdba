"""Top-k entropy estimators (Section 2.1) on the GPU against the oracle.

eti_topk_entropy gives H~ (entropy of p renormalised on the top k), the tail
mass 1 - m and the tail-corrected H^ for every row, through the C ABI.  Same
seeded logits on both sides; tolerances: H~ and H^ 1e-4 relative (1e-6
absolute below 1e-2), tail mass 1e-4 relative or 1e-9 absolute.  The top-k
set is decided on the raw fp32 logits on both sides (the same order), so no
near-tie rule is needed: tokens tied at the k-th value contribute equally.
"""
import math

import numpy as np
import pytest
import torch

import oracle
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


def _run(eti, logits, T, k, V=None):
    B = logits.shape[0]
    f32 = torch.float32
    Ht = torch.full((B,), -7.0, dtype=f32, device=DEV)
    Hh = torch.full((B,), -7.0, dtype=f32, device=DEV)
    tm = torch.full((B,), -7.0, dtype=f32, device=DEV)
    err = torch.full((B,), -7, dtype=torch.int32, device=DEV)
    eti.eti_topk_entropy(logits, T, k, Ht, Hh, err, tail_mass=tm, V=V)
    torch.cuda.synchronize()
    return dict(H_tilde=Ht.cpu().numpy(), H_hat=Hh.cpu().numpy(), tail_mass=tm.cpu().numpy(),
                err=err.cpu().numpy().view(np.uint32))


def _compare(g, r):
    assert np.array_equal(g["err"], r["err"])
    ok = r["err"] == 0
    assert np.isnan(g["H_hat"][~ok]).all() and np.isnan(g["H_tilde"][~ok]).all()
    for key in ("H_tilde", "H_hat"):
        x, y = g[key][ok].astype(np.float64), r[key][ok]
        tol = np.where(y < 1e-2, 1e-6, 1e-4 * y)
        assert (np.abs(x - y) <= tol).all(), (key, float(np.max(np.abs(x - y) / np.maximum(y, 1e-12))))
    x, y = g["tail_mass"][ok].astype(np.float64), r["tail_mass"][ok]
    assert (np.abs(x - y) <= np.maximum(1e-4 * y, 1e-9)).all()
    return float(np.max(np.abs(g["H_hat"][ok] - r["H_hat"][ok]))) if ok.any() else 0.0


@pytest.mark.parametrize("name,ks", [("tiny", (1, 50, 4096, 5000)), ("llama3_8b", (1, 20, 64, 1000)),
                                     ("mixed_batch", (64,))])
def test_topk_entropy_workloads(eti, name, ks):
    w = workloads.WORKLOADS[name]
    if name == "mixed_batch":
        w = w.scaled(B=64)
    lg = workloads.make_logits(w, DEV)
    z, T = lg["logits"], lg["T_in"]
    for k in ks:
        g = _run(eti, z, T, k)
        r = oracle.topk_entropy(z.cpu().numpy(), T.cpu().numpy(), k)
        print(name, k, _compare(g, r))


@pytest.mark.parametrize("B,V,pad", [(1, 1, 0), (3, 2, 1), (5, 7, 3), (2, 1000, 0), (4, 4097, 3),
                                     (6, 50001, 1)])
def test_topk_entropy_ragged_and_unaligned(eti, B, V, pad):
    rng = np.random.default_rng(V + B)
    ld = V + pad
    z = (rng.standard_normal((B, ld)) * rng.uniform(0.2, 6.0, (B, 1))).astype(np.float32)
    T = rng.uniform(0.5, 2.0, B).astype(np.float32)
    if pad:
        # row-major [B, ld] starting 4 bytes past an aligned address: the scalar path
        flat = torch.zeros(B * ld + 1, device=DEV)
        flat[1:] = torch.from_numpy(z).reshape(-1).to(DEV)
        zt = flat[1:].view(B, ld)
    else:
        zt = torch.from_numpy(z).to(DEV)
    Tt = torch.from_numpy(T).to(DEV)
    for k in sorted({1, 2, max(1, V // 3), V, V + 4}):
        g = _run(eti, zt, Tt, k, V=V)
        r = oracle.topk_entropy(z, T, k, V=V)
        _compare(g, r)


def test_topk_entropy_ties_at_the_kth_value(eti):
    """Repeated values straddling the k-th position, ties at the max, -inf
    entries inside K (fewer finite logits than k)."""
    B, V = 6, 3000
    rng = np.random.default_rng(11)
    z = rng.standard_normal((B, V)).astype(np.float32)
    z[0, 100:400] = 1.5                      # 300 ties around the top
    z[1, :] = np.round(z[1, :] * 4) / 4      # many values repeated
    z[2, 5:9] = z[2].max() + 1.0             # four tokens at the max
    z[3, 10:] = -np.inf                      # 10 finite tokens only
    z[4, :] = 0.25                           # uniform row
    z[5, :] = -np.inf
    z[5, 7] = 3.0                            # one finite token
    T = np.ones(B, np.float32)
    zt, Tt = torch.from_numpy(z).to(DEV), torch.from_numpy(T).to(DEV)
    for k in (1, 2, 3, 4, 5, 50, 250, 2999, 3000):
        _compare(_run(eti, zt, Tt, k), oracle.topk_entropy(z, T, k))


def test_topk_entropy_error_rows(eti):
    z = np.random.default_rng(1).standard_normal((5, 700)).astype(np.float32)
    z[0, 3] = np.nan
    z[1, 600] = np.inf
    z[2] = -np.inf
    T = np.array([1, 1, 1, 0, 1], np.float32)
    g = _run(eti, torch.from_numpy(z).to(DEV), torch.from_numpy(T).to(DEV), 10)
    r = oracle.topk_entropy(z, T, 10)
    _compare(g, r)
    assert list(g["err"]) == [oracle.ERR_NONFINITE, oracle.ERR_NONFINITE, oracle.ERR_ALL_NEG_INF,
                              oracle.ERR_BAD_TEMP, 0]
