"""Seeded synthetic inputs for the entropic-time decode step.

This module only draws random inputs with the shapes and value distributions
of the serving workloads the paper targets (Llama-3-shaped GQA layers, a
128,256-token vocabulary, paged KV caches); it holds none of the method's
arithmetic.  Both the CUDA path (through the tests and the benchmark) and the
fp64 oracle read the tensors it makes.

Recipe (per workload):
  * logits  z[b, :] = s_b * N(0, 1), s_b log-uniform on [0.1, 10]; 0-3 token
    ids (count uniform on {0,1,2,3}) get +8.  In the large-batch mixed
    workload every even row instead gets one token at +20 (near-deterministic).
  * H_prev ~ U[0, log V]; H_target = f * log V (f = 0.5 unless swept);
    T_in = 1; tau_in = 0.
  * q, K, V ~ N(0, 1) rounded to bf16; a fraction of the (sequence, kv head,
    block) key chunks is scaled by 4 ("high-norm blocks").
  * context lengths drawn per sequence (uniform or log-uniform, or a fixed
    list), block tables filled from a random permutation of the page pool.
    Pages past a sequence's last block hold -1 in the block table.
Host-side structure uses numpy PCG64(seed); bulk tensors use a torch
generator seeded from the same seed on the requested device.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    Hq: int
    Hkv: int
    D: int
    P: int
    V: int
    ctx: tuple            # ("list", [...]) | ("uniform", lo, hi) | ("loguniform", lo, hi)
    seed: int
    hi_frac: float = 0.0  # fraction of key chunks scaled x4
    spike: float = 8.0
    even_row_spike: float | None = None  # one token at this value on even rows
    pool: int | None = None              # page-pool size (None: exactly the pages used)
    H_target_frac: float = 0.5
    notes: str = ""

    @property
    def max_blocks(self) -> int:
        hi = max(self.ctx[1]) if self.ctx[0] == "list" else self.ctx[2]
        return -(-hi // self.P)

    def scaled(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    # tiny decode step: 4 sequences, MHA 8/8, head_dim 64, page 16, V = 4096
    "tiny": Workload("tiny", B=4, Hq=8, Hkv=8, D=64, P=16, V=4096,
                     ctx=("list", [64, 128, 192, 256]), seed=0),
    # Llama-3-8B-shaped layer step
    "llama3_8b": Workload("llama3_8b", B=64, Hq=32, Hkv=8, D=128, P=16, V=128256,
                          ctx=("uniform", 1024, 8192), seed=1, hi_frac=0.05),
    # long-context step
    "long_ctx": Workload("long_ctx", B=8, Hq=32, Hkv=8, D=128, P=16, V=128256,
                         ctx=("uniform", 32768, 131072), seed=2, hi_frac=0.02),
    # large-batch mixed step, pages scattered over a 2M-page pool
    "mixed_batch": Workload("mixed_batch", B=256, Hq=32, Hkv=8, D=128, P=32, V=128256,
                            ctx=("loguniform", 128, 16384), seed=3, hi_frac=0.05,
                            even_row_spike=20.0, pool=1 << 21),
    # Llama-3-70B-shaped layer step
    "llama3_70b": Workload("llama3_70b", B=128, Hq=64, Hkv=8, D=128, P=16, V=128256,
                           ctx=("uniform", 2048, 32768), seed=4, hi_frac=0.05),
}


def ctx_lengths(w: Workload) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(w.seed))
    kind = w.ctx[0]
    if kind == "list":
        L = np.array(w.ctx[1], dtype=np.int64)
        assert len(L) == w.B
    elif kind == "uniform":
        L = rng.integers(w.ctx[1], w.ctx[2] + 1, size=w.B)
    elif kind == "loguniform":
        L = np.exp(rng.uniform(math.log(w.ctx[1]), math.log(w.ctx[2]), size=w.B))
        L = np.clip(np.round(L), w.ctx[1], w.ctx[2]).astype(np.int64)
    else:
        raise ValueError(kind)
    return L.astype(np.int32)


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def make_logits(w: Workload, device="cpu", ld: int | None = None) -> dict:
    """Logits and per-sequence controller state for one decode step."""
    rng = np.random.Generator(np.random.PCG64(w.seed + 1000))
    B, V = w.B, w.V
    ld = V if ld is None else ld
    scale = np.exp(rng.uniform(math.log(0.1), math.log(10.0), size=B)).astype(np.float32)
    z = torch.empty((B, ld), dtype=torch.float32, device=device)
    g = _gen(device, w.seed + 2000)
    for b in range(B):
        z[b, :V].normal_(generator=g)
    z[:, :V] *= torch.from_numpy(scale).to(device)[:, None]
    if ld > V:
        z[:, V:] = float("nan")  # never read: columns past V
    for b in range(B):
        if w.even_row_spike is not None and b % 2 == 0:
            z[b, int(rng.integers(0, V))] += w.even_row_spike
        else:
            n = min(int(rng.integers(0, 4)), V)
            for x in rng.choice(V, size=n, replace=False):
                z[b, int(x)] += w.spike
    logV = math.log(V)
    H_prev = torch.from_numpy(rng.uniform(0.0, logV, size=B).astype(np.float32)).to(device)
    H_target = torch.full((B,), w.H_target_frac * logV, dtype=torch.float32, device=device)
    T_in = torch.ones(B, dtype=torch.float32, device=device)
    tau = torch.zeros(B, dtype=torch.float32, device=device)
    return dict(logits=z, H_prev=H_prev, H_target=H_target, T_in=T_in, tau=tau, V=V, ld=ld)


def make_kv(w: Workload, device="cpu", pool: int | None = None, poison_tail: bool = False,
            chunk_pages: int = 4096) -> dict:
    """q, paged K/V caches, block table and context lengths for one layer step.

    Only the pages that some sequence references are written; the rest of the
    pool is left as allocated.  poison_tail=True fills the token slots past
    each sequence's length in its last page with NaN (they must never reach
    a result).
    """
    rng = np.random.Generator(np.random.PCG64(w.seed + 3000))
    L = ctx_lengths(w)
    nb = (L + w.P - 1) // w.P
    total = int(nb.sum())
    pool = pool or w.pool or total
    pool = max(pool, total)
    page_ids = rng.permutation(pool)[:total].astype(np.int64)
    mb = w.max_blocks
    bt = np.full((w.B, mb), -1, dtype=np.int32)
    owner = np.empty(total, dtype=np.int64)       # sequence of each used page
    pos = 0
    for b in range(w.B):
        bt[b, :nb[b]] = page_ids[pos:pos + nb[b]]
        owner[pos:pos + nb[b]] = b
        pos += nb[b]
    # high-norm key chunks: Bernoulli(hi_frac) per (page, kv head)
    hi = rng.random((total, w.Hkv)) < w.hi_frac if w.hi_frac > 0 else np.zeros((total, w.Hkv), bool)

    q = torch.empty((w.B, w.Hq, w.D), dtype=torch.float32, device=device)
    q.normal_(generator=_gen(device, w.seed + 4000))
    q = q.to(torch.bfloat16)
    k_cache = torch.empty((pool, w.Hkv, w.P, w.D), dtype=torch.bfloat16, device=device)
    v_cache = torch.empty((pool, w.Hkv, w.P, w.D), dtype=torch.bfloat16, device=device)
    gk = _gen(device, w.seed + 5000)
    gv = _gen(device, w.seed + 6000)
    hi_t = torch.from_numpy(hi).to(device)
    ids_t = torch.from_numpy(page_ids).to(device)
    for s in range(0, total, chunk_pages):
        e = min(total, s + chunk_pages)
        kc = torch.empty((e - s, w.Hkv, w.P, w.D), dtype=torch.float32, device=device)
        kc.normal_(generator=gk)
        kc = torch.where(hi_t[s:e, :, None, None], kc * 4.0, kc)
        k_cache.index_copy_(0, ids_t[s:e], kc.to(torch.bfloat16))
        vc = torch.empty_like(kc)
        vc.normal_(generator=gv)
        v_cache.index_copy_(0, ids_t[s:e], vc.to(torch.bfloat16))
        del kc, vc
    if poison_tail:
        for b in range(w.B):
            r = int(L[b]) % w.P
            if nb[b] > 0 and r:
                pg = int(bt[b, nb[b] - 1])
                k_cache[pg, :, r:, :] = float("nan")
                v_cache[pg, :, r:, :] = float("nan")
    return dict(q=q, k_cache=k_cache, v_cache=v_cache,
                block_table=torch.from_numpy(bt).to(device),
                ctx_lens=torch.from_numpy(L).to(device),
                num_pages=pool, scale=1.0 / math.sqrt(w.D), hi_chunks=hi, page_ids=page_ids,
                owner=owner)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """The 16-bit patterns of a bf16 tensor as a host uint16 array."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def gather_sequences(kv: dict, seqs) -> dict:
    """A compact host copy of the pages of the given sequences, with the block
    table rewritten to index it (for spot checks of large workloads)."""
    seqs = [int(s) for s in seqs]
    bt = kv["block_table"][seqs].cpu().numpy()
    L = kv["ctx_lens"][seqs].cpu().numpy()
    P = kv["k_cache"].shape[2]
    used = []
    new_bt = np.full_like(bt, -1)
    for i, b in enumerate(seqs):
        n = (int(L[i]) + P - 1) // P
        for j in range(n):
            new_bt[i, j] = len(used)
            used.append(int(bt[i, j]))
    idx = torch.tensor(used, dtype=torch.long, device=kv["k_cache"].device)
    kc = kv["k_cache"].index_select(0, idx) if used else kv["k_cache"][:0]
    vc = kv["v_cache"].index_select(0, idx) if used else kv["v_cache"][:0]
    return dict(q=bf16_bits(kv["q"][seqs]), k_cache=bf16_bits(kc), v_cache=bf16_bits(vc),
                block_table=new_bt.astype(np.int32), ctx_lens=L.astype(np.int32),
                num_pages=len(used), scale=kv["scale"], pages=np.asarray(used, np.int64))
