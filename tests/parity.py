"""Shared comparison logic for the GPU-vs-oracle parity tests.

Tolerances (stated here once, used by every parity test):
  * entropy H: 1e-4 relative, or 1e-6 nats absolute when H < 1e-2;
  * temperature T_out, entropy flow dH, tau: 1e-4 relative (dH and tau also
    1e-5 absolute, since dH can cancel to ~0);
  * theta_next: 2e-4 absolute (it is 1 - H / log V, an O(1) quantity whose
    error is the H error divided by log V);
  * surprisal: 1e-4 relative or 1e-5 absolute;
  * sampled token: exact, unless the oracle's Gumbel-max key of the GPU's
    token is within 1e-5 of the best key (counted as a tie and reported);
  * keep mask / kept lists: exact, unless the oracle's block score is within
    1e-5 * max(1, theta) of theta, or within 1e-5 * max(1, s_k) of the k-th
    best score at the B_min boundary (counted as ties); no wider band;
  * block scores (no bound is stated for them): within 2e-5 * max(1, |score|)
    plus the block's fp32 evaluation band (score_bands);
  * attention output (bf16 from fp32 accumulation over bf16 K/V): 2e-2
    absolute.
Every comparison adds its counts to TALLY, which the session prints at the end
(tests/conftest.py), and the tie counts are capped: at most
max(2, 1e-4 * compared) ties per call.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads

H_REL, H_ABS_SMALL = 1e-4, 1e-6
KEY_TIE = 1e-5
MASK_TIE = 1e-5
ATTN_ABS = 2e-2
TIE_CAP = 1e-4

# counts over the whole session (printed by the terminal summary hook)
TALLY = dict(token_rows=0, token_ties=0, worst_token_gap=0.0, mask_block_heads=0, mask_ties=0,
             score_block_heads=0, worst_score_err=0.0, attn_seqs=0, worst_attn_err=0.0)


def tie_cap(compared: int) -> int:
    return max(2, int(TIE_CAP * compared))


def tally_line() -> str:
    t = TALLY
    return (f"parity tally: sampled tokens {t['token_rows']} rows, {t['token_ties']} Gumbel near-ties "
            f"(worst key gap {t['worst_token_gap']:.2e}); keep masks {t['mask_block_heads']} block-heads, "
            f"{t['mask_ties']} near-ties within 1e-5; block scores {t['score_block_heads']} block-heads, "
            f"worst error {t['worst_score_err']:.2e} (relative to max(1, |score|)); attention "
            f"{t['attn_seqs']} sequences, worst |error| {t['worst_attn_err']:.2e}")


def run_ets(eti, lg: dict, params=None, seed=0, offset=0, V=None, theta_prev=None):
    """Run eti_entropy_temp_sample on the workload's logits; numpy results.
    theta_prev (numpy [B]) fills theta_next first (read by the dtheta guard)."""
    B = lg["logits"].shape[0]
    dev = lg["logits"].device
    f32, i32 = torch.float32, torch.int32
    tau = lg["tau"].clone()
    out = dict(tok=torch.empty(B, dtype=i32, device=dev), H=torch.empty(B, dtype=f32, device=dev),
               T_out=torch.empty(B, dtype=f32, device=dev), dH=torch.empty(B, dtype=f32, device=dev),
               theta_next=(torch.empty(B, dtype=f32, device=dev) if theta_prev is None else
                           torch.tensor(np.asarray(theta_prev, np.float32), device=dev)),
               surprisal=torch.empty(B, dtype=f32, device=dev),
               err=torch.empty(B, dtype=i32, device=dev))
    ws = torch.empty(eti.entropy_temp_sample_workspace_size(B, V or lg["logits"].shape[1]),
                     dtype=torch.uint8, device=dev)
    eti.eti_entropy_temp_sample(lg["logits"], lg["T_in"], lg["H_prev"], tau, lg["H_target"],
                                out["tok"], out["H"], out["T_out"], out["err"], ws, params=params,
                                seed=seed, offset=offset, dH=out["dH"],
                                theta_next=out["theta_next"], tok_surprisal=out["surprisal"], V=V)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["tau"] = tau.cpu().numpy()
    res["err"] = res["err"].view(np.uint32)
    return res


def oracle_ets(lg: dict, ctrl=None, seed=0, offset=0, V=None, theta_prev=None):
    return oracle.entropy_temp_sample(lg["logits"].cpu().numpy(), lg["T_in"].cpu().numpy(),
                                      lg["H_prev"].cpu().numpy(), lg["tau"].cpu().numpy(),
                                      lg["H_target"].cpu().numpy(), ctrl, seed=seed, offset=offset,
                                      V=V, theta_prev=theta_prev)


def _close(a, b, rel, abs_=0.0):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return np.abs(a - b) <= np.maximum(rel * np.abs(b), abs_)


def compare_ets(gpu: dict, ref: dict, lg: dict, seed=0, offset=0, V=None) -> dict:
    """Assert parity of every output of the entropy/sample call; return tie stats."""
    ok_rows = ref["err"] == 0
    assert np.array_equal(gpu["err"], ref["err"]), (gpu["err"], ref["err"])
    bad = ~ok_rows
    assert (gpu["tok"][bad] == -1).all() and np.isnan(gpu["H"][bad]).all()
    Hr, Hg = ref["H"][ok_rows], gpu["H"][ok_rows].astype(np.float64)
    small = Hr < 1e-2
    okH = np.where(small, np.abs(Hg - Hr) <= H_ABS_SMALL, np.abs(Hg - Hr) <= H_REL * Hr)
    assert okH.all(), f"H mismatch: worst rel {np.max(np.abs(Hg - Hr) / np.maximum(Hr, 1e-12))}"
    assert _close(gpu["T_out"][ok_rows], ref["T_out"][ok_rows], 1e-4).all()
    assert _close(gpu["dH"][ok_rows], ref["dH"][ok_rows], 1e-4, 1e-5).all()
    assert _close(gpu["tau"][ok_rows], ref["tau"][ok_rows], 1e-4, 1e-5).all()
    assert _close(gpu["theta_next"][ok_rows], ref["theta_next"][ok_rows], 0.0, 2e-4).all()
    assert (gpu["tau"][bad] == lg["tau"].cpu().numpy()[bad]).all()
    # sampled tokens: exact except Gumbel near-ties
    z = lg["logits"].cpu().numpy()
    T = lg["T_in"].cpu().numpy()
    ties, worst = 0, 0.0
    for b in np.nonzero(ok_rows)[0]:
        if gpu["tok"][b] == ref["tok"][b]:
            continue
        Vb = z.shape[1] if V is None else V
        kg = oracle.sample_key(z[b, :Vb], float(T[b]), seed, offset, int(b), int(gpu["tok"][b]))
        kb = oracle.sample_key(z[b, :Vb], float(T[b]), seed, offset, int(b), int(ref["tok"][b]))
        gap = kb - kg
        worst = max(worst, gap)
        assert gap < KEY_TIE, f"row {b}: GPU token {gpu['tok'][b]} vs oracle {ref['tok'][b]}, key gap {gap}"
        ties += 1
    sr, sg = ref["surprisal"][ok_rows], gpu["surprisal"][ok_rows]
    same = gpu["tok"][ok_rows] == ref["tok"][ok_rows]
    assert _close(sg[same], sr[same], 1e-4, 1e-5).all()
    rows = int(ok_rows.sum())
    assert ties <= tie_cap(rows), f"{ties} token near-ties in {rows} rows"
    TALLY["token_rows"] += rows
    TALLY["token_ties"] += ties
    TALLY["worst_token_gap"] = max(TALLY["worst_token_gap"], worst)
    return dict(rows=rows, token_ties=ties, worst_tie_gap=worst)


# ---------------------------------------------------------------------------
def host_kv(kv: dict) -> dict:
    return dict(q=workloads.bf16_bits(kv["q"]), k=workloads.bf16_bits(kv["k_cache"]),
                v=workloads.bf16_bits(kv["v_cache"]), bt=kv["block_table"].cpu().numpy(),
                L=kv["ctx_lens"].cpu().numpy(), scale=kv["scale"], num_pages=kv["num_pages"])


def host_from_gather(sub: dict) -> dict:
    """workloads.gather_sequences output in the host_kv layout."""
    return dict(q=sub["q"], k=sub["k_cache"], v=sub["v_cache"], bt=sub["block_table"],
                L=sub["ctx_lens"], scale=sub["scale"], num_pages=sub["num_pages"],
                pages=sub["pages"])


def score_bands(ref: dict, n: dict, score_mode: int = 0) -> np.ndarray:
    """Per (sequence, kv head, block) bound on |Ibar_gpu - Ibar_exact| from fp32 scores.

    The kernel forms x_i = s q.k_i as an fp32 dot product of D bf16 products,
    error |dx| <= c sqrt(D) 2^-24 s |q| |k_i| with c = 4 (the root-D growth of
    rounding errors with a margin; the worst-case D 2^-24 bound is far looser).
    Then |da_i / a_i| <= 2 |dx| and, from I_b = sum a_i (-log a_i) and
    H = sum_b I_b,  |dIbar_b| / Ibar_b <= 2 |dx| ((I_b + A_b) / I_b + (H + 1) / H),
    A_b the block's attention mass: the bound is large exactly where one token
    takes nearly all of a block's attention (I_b << A_b).  In modes E and M the
    per-token weight does not depend on a_i (s_i >= 0 or 1), so the numerator
    and the normaliser each move by at most 2 |dx| relative: 4 |dx| in all.
    """
    q = (n["q"].astype(np.uint32) << 16).view(np.float32)           # [B, Hq, D]
    k = (n["k"].astype(np.uint32) << 16).view(np.float32)           # [pages, Hkv, P, D]
    B, Hq, D = q.shape
    _, Hkv, P, _ = k.shape
    g = Hq // Hkv
    mb = n["bt"].shape[1]
    band = np.zeros((B, Hkv, mb))
    knorm = np.empty(k.shape[:3])                                    # [pages, Hkv, P]
    with np.errstate(invalid="ignore", over="ignore"):
        for p0 in range(0, k.shape[0], 4096):                        # bounded temporaries
            kk = k[p0:p0 + 4096].astype(np.float64)
            knorm[p0:p0 + 4096] = np.sqrt(np.einsum("...d,...d->...", kk, kk))
    for b in range(B):
        L = int(n["L"][b])
        nb = -(-L // P) if L > 0 else 0
        if nb == 0:
            continue
        pages = n["bt"][b, :nb]
        if (pages < 0).any() or (pages >= k.shape[0]).any():
            continue
        valid = np.arange(nb * P).reshape(nb, P) < L
        for kvh in range(Hkv):
            kn = np.where(valid, knorm[pages, kvh], 0.0).max()
            qn = np.linalg.norm(q[b, kvh * g:(kvh + 1) * g].astype(np.float64), axis=-1).max()
            dx = 4.0 * np.sqrt(D) * 2.0 ** -24 * n["scale"] * qn * kn
            for hh in range(g):
                h = kvh * g + hh
                I = ref["head_I"][b, h, :nb]
                A = ref["head_A"][b, h, :nb]
                H = ref["head_H"][b, h]
                if H <= 0:
                    continue
                if score_mode == 0:
                    kappa = (I + A) / np.maximum(I, 1e-300) + (H + 1.0) / H
                else:
                    kappa = 2.0
                nrm = nb * I / H
                band[b, kvh, :nb] = np.maximum(band[b, kvh, :nb], 2.0 * dx * kappa * nrm)
    return band


def compare_masks(gpu_mask, gpu_idx, gpu_cnt, ref: dict, theta, B_min, P, L, band=None) -> dict:
    """Keep sets equal except for near-threshold / near-budget-boundary ties.

    A block may differ only if its oracle score is within 1e-5 max(1, |theta|)
    of theta, or within 1e-5 max(1, |s_k|) of the k-th best score s_k at the
    B_min boundary.  `band` (score_bands) is only quoted in the failure
    message, to tell an ill-conditioned score from a wrong one."""
    B, Hkv, mb = ref["keep_mask"].shape
    band = np.zeros((B, Hkv, mb)) if band is None else band
    ties = 0
    compared = 0
    for b in range(B):
        n = -(-int(L[b]) // P) if L[b] > 0 else 0
        th = float(theta[b])
        for h in range(Hkv):
            gm, rm = gpu_mask[b, h, :n].astype(bool), ref["keep_mask"][b, h, :n].astype(bool)
            compared += n
            assert not gpu_mask[b, h, n:].any()
            c = int(gpu_cnt[b, h])
            assert c == int(gm.sum())
            assert np.array_equal(gpu_idx[b, h, :c], np.nonzero(gm)[0])
            assert (gpu_idx[b, h, c:] == -1).all()
            diff = np.nonzero(gm != rm)[0]
            if len(diff) == 0:
                continue
            s = ref["block_score"][b, h, :n]
            k = min(max(B_min, 0), n)
            order = np.argsort(-s, kind="stable")
            sk = s[order[k - 1]] if 0 < k < n else None
            for j in diff:
                near_th = np.isfinite(th) and abs(s[j] - th) <= MASK_TIE * max(1.0, abs(th))
                near_k = sk is not None and abs(s[j] - sk) <= MASK_TIE * max(1.0, abs(sk))
                assert near_th or near_k, (f"seq {b} kvh {h} block {j}: gpu {gm[j]} oracle {rm[j]} "
                                           f"score {s[j]} theta {th} s_k {sk} "
                                           f"(fp32 evaluation band of the score {band[b, h, j]:.3g})")
                ties += 1
    assert ties <= tie_cap(compared), f"{ties} keep-mask near-ties in {compared} block-heads"
    TALLY["mask_block_heads"] += compared
    TALLY["mask_ties"] += ties
    return dict(mask_ties=ties, block_heads=compared)


def compare_scores(gpu_score, ref_score, P, L, band=None):
    """Block scores within 2e-5 relative plus the fp32 evaluation band."""
    B, Hkv, mb = ref_score.shape
    band = np.zeros((B, Hkv, mb)) if band is None else band
    worst = 0.0
    for b in range(B):
        n = -(-int(L[b]) // P) if L[b] > 0 else 0
        if not n:
            continue
        g, r = gpu_score[b, :, :n].astype(np.float64), ref_score[b, :, :n]
        err = np.abs(g - r)
        tol = 2e-5 * np.maximum(1.0, np.abs(r)) + band[b, :, :n]
        assert (err <= tol).all(), (b, np.unravel_index(np.argmax(err - tol), err.shape),
                                    float((err - tol).max()))
        worst = max(worst, float(np.max(err / np.maximum(1.0, np.abs(r)))))
        TALLY["score_block_heads"] += int(err.size)
    TALLY["worst_score_err"] = max(TALLY["worst_score_err"], worst)
    return worst


def compare_attention(gpu_out, ref_out, rows=None):
    g = gpu_out.astype(np.float64)
    err = np.abs(g - ref_out)
    assert np.isfinite(g).all()
    worst = float(err.max()) if err.size else 0.0
    assert worst < ATTN_ABS, worst
    TALLY["attn_seqs"] += int(g.shape[0]) if g.ndim == 3 else 0
    TALLY["worst_attn_err"] = max(TALLY["worst_attn_err"], worst)
    return worst
