"""Seeded synthetic inputs shaped like the SAS workloads.

This module only draws random numbers: it holds none of the method's
arithmetic, and both the CUDA path and the oracle take their inputs from it.
Everything is drawn in float32 on the CPU with a seeded torch generator and
then rounded to the storage dtype (bf16 for activations and weights, fp32 for
scores), so that every consumer sees the same bits.

Score regimes (the paper does not describe how coherent the selections of
neighbouring queries are, so the benchmark names three):
  R1  block-coherent scores: s[i, m] = u[floor(i / b), m] + 0.05 eps[i, m]
  R2  block-correlated queries for the learned-selector path:
      q_i = (mu[floor(i / b)] + 0.3 eps_i) / sqrt(1.09), marginally N(0, 1)
  R3  independent scores: s ~ N(0, 1)
"""
from __future__ import annotations

import math

import torch


def _gen(seed):
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def normal(shape, seed, std=1.0):
    """float32 N(0, std^2) tensor on the CPU."""
    return torch.randn(*shape, generator=_gen(seed), dtype=torch.float32) * std


def qkv(B, H, N, d, seed=0, regime="iid", block=64):
    """Q, K, V as bf16 [B, H, N, d].  regime 'iid' or 'R2' (block-correlated Q)."""
    K = normal((B, H, N, d), seed + 1).to(torch.bfloat16)
    V = normal((B, H, N, d), seed + 2).to(torch.bfloat16)
    if regime == "R2":
        nb = -(-N // block)
        mu = normal((B, H, nb, d), seed + 3)
        eps = normal((B, H, N, d), seed + 4)
        idx = torch.arange(N) // block
        Q = (mu[:, :, idx, :] + 0.3 * eps) / math.sqrt(1.09)
        Q = Q.to(torch.bfloat16)
    else:
        Q = normal((B, H, N, d), seed).to(torch.bfloat16)
    return Q, K, V


def scores(B, H, N, C, seed=0, regime="R1", block=64):
    """Selector scores as fp32 [B, H, N, C].  regime 'R1' (block-coherent) or 'R3' (iid)."""
    if regime == "R1":
        nb = -(-N // block)
        u = normal((B, H, nb, C), seed + 10)
        eps = normal((B, H, N, C), seed + 11)
        idx = torch.arange(N) // block
        return (u[:, :, idx, :] + 0.05 * eps).contiguous()
    return normal((B, H, N, C), seed + 12)


def integer_scores(B, H, N, C, seed=0, levels=4):
    """Small-integer fp32 scores: many exact ties, for the tie rule."""
    g = _gen(seed + 20)
    return torch.randint(0, levels, (B, H, N, C), generator=g).to(torch.float32)


def integer_selector_inputs(B, H, N, d, d_sel, seed=0, nnz=4):
    """Q, K with integer entries in [-3, 3], V ~ N(0, 1), and sparse selector
    projections with entries in {-1, 0, 1} (nnz non-zeros per output row).

    With these inputs every sum the learned selector forms is exactly
    representable in fp32, so any two correct implementations see identical
    scores (and identical ties)."""
    g = _gen(seed + 50)
    Q = torch.randint(-3, 4, (B, H, N, d), generator=g).to(torch.bfloat16)
    K = torch.randint(-3, 4, (B, H, N, d), generator=g).to(torch.bfloat16)
    V = normal((B, H, N, d), seed + 51).to(torch.bfloat16)
    W = []
    for _ in range(2):
        w = torch.zeros(H, d_sel, d)
        cols = torch.stack([torch.randperm(d, generator=g)[:nnz] for _ in range(H * d_sel)]).view(H, d_sel, nnz)
        sign = torch.randint(0, 2, (H, d_sel, nnz), generator=g).float() * 2 - 1
        w.scatter_(2, cols, sign)
        W.append(w.to(torch.bfloat16))
    return Q, K, V, W[0], W[1]


def selector_weights(H, d, d_sel, seed=0, std=0.02):
    """Wq, Wk as bf16 [H, d_sel, d] (linear-layer layout [out, in])."""
    Wq = normal((H, d_sel, d), seed + 30, std).to(torch.bfloat16)
    Wk = normal((H, d_sel, d), seed + 31, std).to(torch.bfloat16)
    return Wq, Wk


def mlp(T, D, F, seed=0, std=0.02, bias=False):
    """X [T, D], W1 [F, D], W2 [D, F] (and b1 [F], b2 [D] if bias) as bf16."""
    X = normal((T, D), seed + 40).to(torch.bfloat16)
    W1 = normal((F, D), seed + 41, std).to(torch.bfloat16)
    W2 = normal((D, F), seed + 42, std).to(torch.bfloat16)
    if not bias:
        return X, W1, W2, None, None
    b1 = normal((F,), seed + 43, std).to(torch.bfloat16)
    b2 = normal((D,), seed + 44, std).to(torch.bfloat16)
    return X, W1, W2, b1, b2


# ------------------------------------------------------------------ decode

def _dev_normal(shape, seed, device, std=1.0):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return torch.randn(*shape, generator=g, device=device, dtype=torch.float32) * std


def decode_layout(lens, max_blocks, seed=0, spare_pages=3, block=64):
    """Page assignment of a paged decode cache.

    lens: tokens each sequence will hold.  Every sequence gets ceil(len/64)
    pages out of a seeded permutation of P = sum + spare_pages pages; block
    table entries past a sequence's last page are -1.  Returns (block_table
    int32 [B, max_blocks], P)."""
    need = [-(-int(n) // block) for n in lens]
    P = sum(need) + spare_pages
    perm = torch.randperm(P, generator=_gen(seed + 60))
    table = torch.full((len(lens), max_blocks), -1, dtype=torch.int32)
    k = 0
    for bi, c in enumerate(need):
        table[bi, :c] = perm[k:k + c].to(torch.int32)
        k += c
    return table, P


def decode_cache(P, Hkv, d, seed=0, device="cpu", exact=False, block=64):
    """K, V pages [P, Hkv, 64, d] as bf16.  Keys are block-coherent,
    k = (mu_page + 0.5 eps) / sqrt(1.25), so block summaries differ from block
    to block; values N(0, 1).  exact=True: keys are integers in [-3, 3]."""
    if exact:
        g = torch.Generator(device=device)
        g.manual_seed(int(seed + 70))
        K = torch.randint(-3, 4, (P, Hkv, block, d), generator=g, device=device).to(torch.bfloat16)
    else:
        mu = _dev_normal((P, Hkv, 1, d), seed + 71, device)
        K = ((mu + 0.5 * _dev_normal((P, Hkv, block, d), seed + 72, device)) / math.sqrt(1.25)).to(torch.bfloat16)
    V = _dev_normal((P, Hkv, block, d), seed + 73, device).to(torch.bfloat16)
    return K, V


def decode_queries(B, Hq, Hkv, d, seed=0, device="cpu", exact=False):
    """q [B, Hq, d], k_new and v_new [B, Hkv, d] as bf16 (integers in [-3, 3]
    for q and k_new when exact)."""
    if exact:
        g = torch.Generator(device=device)
        g.manual_seed(int(seed + 80))
        q = torch.randint(-3, 4, (B, Hq, d), generator=g, device=device).to(torch.bfloat16)
        kn = torch.randint(-3, 4, (B, Hkv, d), generator=g, device=device).to(torch.bfloat16)
    else:
        q = _dev_normal((B, Hq, d), seed + 81, device).to(torch.bfloat16)
        kn = _dev_normal((B, Hkv, d), seed + 82, device).to(torch.bfloat16)
    vn = _dev_normal((B, Hkv, d), seed + 83, device).to(torch.bfloat16)
    return q, kn, vn


def decode_selector_weights(Hkv, G, d, d_sel, seed=0, device="cpu", exact=False, std=0.02, nnz=4):
    """Wq [Hkv, d_sel, G*d] and Wk [Hkv, d_sel, d] as bf16; exact=True gives
    sparse {-1, 0, 1} rows with nnz non-zeros."""
    if not exact:
        Wq = _dev_normal((Hkv, d_sel, G * d), seed + 90, device, std).to(torch.bfloat16)
        Wk = _dev_normal((Hkv, d_sel, d), seed + 91, device, std).to(torch.bfloat16)
        return Wq, Wk
    g = _gen(seed + 92)
    out = []
    for width in (G * d, d):
        w = torch.zeros(Hkv, d_sel, width)
        cols = torch.stack([torch.randperm(width, generator=g)[:nnz] for _ in range(Hkv * d_sel)])
        sign = torch.randint(0, 2, (Hkv * d_sel, nnz), generator=g).float() * 2 - 1
        w.view(Hkv * d_sel, width).scatter_(1, cols, sign)
        out.append(w.to(torch.bfloat16).to(device))
    return out[0], out[1]
