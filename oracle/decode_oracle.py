"""Plain fp64 CPU oracle for the SAS decode step (Alg. 2, one new token per sequence).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: only the tests, the smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the CUDA library.

What one decode step computes (Alg. 2; Sec. 5, inference implementation: the
selector scores every cached block, the Top-K blocks are chosen once per query
group, and only those blocks' keys and values are read):

  the new token sits at position i = n - 1 of a cache of n tokens, its own key
  and value included.  For each KV head (a group of G query heads sharing keys
  and values):
    q~    = bf16(Wq_g [q_0; q_1; ...; q_{G-1}])       gate query of the group
    K~_m  = bf16(Wk_g mean(K_Bm)),  m < C = floor(i / b)   block summaries (App. B)
    s_m   = q~ . K~_m / sqrt(d_s)                     (Alg. 2 step 1)
    I     = TopK(s, K)                                (Alg. 2 step 2)
    S     = B_0 + the blocks of I, B_0 = tokens C*b .. i   (Alg. 2 step 3)
    o_h   = softmax(sm_scale q_h K_S^T) V_S  for every head h of the group (step 4)
  The dense decode it is compared with attends to all tokens 0 .. i.

Readings of points the paper leaves open:

  * Group gate query.  The paper selects per query group but does not say how
    the group's G query vectors form the gate query.  Reading: they are
    concatenated head by head (head 0 first) and projected by one matrix
    Wq_g of shape [d_s, G*d].  With G = 1 this is the prefill selector of the
    library (q~ = bf16(Wq q)); averaging the per-head queries is the special
    case Wq_g = [W, ..., W] / G.
  * Top-K, ties and short histories follow the prefill oracle: exact-K, ties to
    the lower block index, C <= K keeps every historical block.
  * Paged cache: logical block m of sequence b lives in page block_table[b, m];
    a page holds the 64 tokens of one block for every KV head,
    K_cache[page, kv_head, slot, :].
  * Query head h belongs to KV head h // G.

Arrays are float64 numpy arrays holding the bf16-rounded values the GPU sees.
"""
from __future__ import annotations

import math

import numpy as np

from oracle.sas_oracle import block_summaries, round_to_bf16, topk_blocks


def decode_group(q_g, K_ctx, V_ctx, Wq_g, Wk, b, topk, sm_scale=None, dense=False):
    """One decode step of one KV group over a contiguous context.

    q_g:   [G, d] queries of the group's heads for the new token.
    K_ctx, V_ctx: [n, d] keys / values of positions 0 .. n-1 (n >= 1); the new
           token is position n - 1.
    Wq_g:  [d_s, G*d];  Wk: [d_s, d].
    Returns dict with O [G, d], LSE [G] (natural log), sel (ascending block
    indices, length min(K, C)), scores [C], summaries [C, d_s] (the K~_m).
    """
    G, d = q_g.shape
    n = K_ctx.shape[0]
    i = n - 1
    C = i // b
    d_s = Wq_g.shape[0]
    if sm_scale is None:
        sm_scale = 1.0 / math.sqrt(d)
    qt = round_to_bf16(Wq_g @ q_g.reshape(G * d))
    kt = round_to_bf16(block_summaries(K_ctx[:C * b], b) @ Wk.T) if C > 0 else np.zeros((0, d_s))
    s = kt @ qt / math.sqrt(d_s)
    if dense:
        sel = np.arange(C)
    else:
        sel = np.sort(np.asarray(topk_blocks(s, topk), dtype=np.int64))
    keys = np.concatenate([np.arange(m * b, (m + 1) * b) for m in sel] + [np.arange(C * b, n)])
    O = np.zeros((G, V_ctx.shape[1]))
    LSE = np.zeros(G)
    for h in range(G):
        z = sm_scale * (K_ctx[keys] @ q_g[h])
        zmax = z.max()
        w = np.exp(z - zmax)
        O[h] = (w @ V_ctx[keys]) / w.sum()
        LSE[h] = zmax + math.log(w.sum())
    return {"O": O, "LSE": LSE, "sel": sel, "scores": s, "summaries": kt}


def gather_context(cache, block_table_row, n, kv_head, b):
    """Contiguous [n, d] keys (or values) of one sequence and KV head from the paged cache."""
    nb = -(-n // b)
    pages = [cache[int(block_table_row[m]), kv_head] for m in range(nb)]
    return np.concatenate(pages, axis=0)[:n]


def decode_step(q, K_cache, V_cache, block_table, seq_lens, Wq, Wk, b, topk, sm_scale=None, dense=False,
                groups=None):
    """One decode step for a batch of sequences over a paged cache.

    q: [B, Hq, d]; K_cache, V_cache: [P, Hkv, b, d]; block_table: [B, max_blocks]
    int; seq_lens: [B] tokens in the cache including the new one; Wq: [Hkv, d_s,
    G*d]; Wk: [Hkv, d_s, d].  groups: optional list of (batch, kv_head) pairs to
    evaluate (default all).
    Returns dict of O [B, Hq, d], LSE [B, Hq], sel_idx [B, Hkv, K] (ascending,
    -1 padded), and per evaluated group its scores and summaries.
    """
    B, Hq, d = q.shape
    Hkv = K_cache.shape[1]
    G = Hq // Hkv
    O = np.full((B, Hq, d), np.nan)
    LSE = np.full((B, Hq), np.nan)
    sel_idx = np.full((B, Hkv, max(topk, 1)), -1, dtype=np.int64)
    extra = {}
    groups = groups if groups is not None else [(bi, g) for bi in range(B) for g in range(Hkv)]
    for bi, g in groups:
        n = int(seq_lens[bi])
        Kc = gather_context(K_cache, block_table[bi], n, g, b)
        Vc = gather_context(V_cache, block_table[bi], n, g, b)
        r = decode_group(q[bi, g * G:(g + 1) * G], Kc, Vc, Wq[g], Wk[g], b, topk, sm_scale, dense)
        O[bi, g * G:(g + 1) * G] = r["O"]
        LSE[bi, g * G:(g + 1) * G] = r["LSE"]
        if not dense:
            sel_idx[bi, g, :len(r["sel"])] = r["sel"]
        extra[(bi, g)] = r
    return {"O": O, "LSE": LSE, "sel_idx": sel_idx[:, :, :topk], "groups": extra}


def decode_bytes_per_group(n, b, topk, d, d_s, G, dense=False):
    """Algorithmic HBM bytes one decode step moves for one KV group (bf16
    tensors read once, outputs written once): the new token's key and value
    (read, then written into the cache), the gate query weights and the
    queries, the C block summaries, the keys and values of the attended
    tokens, and O."""
    i = n - 1
    C = i // b
    attended = (C if dense else min(topk, C)) * b + (i - C * b + 1)
    by = 4 * 2 * d                        # k_new, v_new read and appended
    by += 2 * (G * d)                     # queries
    if not dense:
        by += 2 * d_s * G * d             # Wq_g
        by += 2 * C * d_s                 # summaries read by the scorer
    by += 2 * 2 * attended * d            # keys and values
    by += 2 * G * d                       # O
    return by
