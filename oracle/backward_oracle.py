"""Plain fp64 CPU oracle for the backward pass of the SAS training forward.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: only the tests, the smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the CUDA library.

What it computes (Alg. 4 of App. E, gradients of Eq. ours_train; App. D for the
gate gradient and the sparse-scope score gradient):

  forward of a row i (gate position inner, softmax gates, training mode):
    z_j  = sm_scale q_i.k_j + log g_{b(j)}   for j in S_i = B_0 + kept blocks
    p    = softmax(z),  o_i = sum_j p_j v_j
  given dO (the loss gradient of O):
    dp_j    = dO_i . v_j,   Delta_i = dO_i . o_i
    dz_j    = p_j (dp_j - Delta_i)                      (softmax backward)
    dQ_i    = sm_scale sum_j dz_j k_j
    dK_j   += sm_scale dz_j q_i,  dV_j += p_j dO_i
    dlogg_m = sum_{j in B_m} dz_j  for every kept historical block m
            (= g_m dg_m with the paper's dg_m = sum_{j in B_m} (p_j / g_m) dO.(v_j - o))
  sparse-scope score gradient (App. D, training scope; the Top-K choice is a
  constant of the forward):
    ds_m = dlogg_m [m kept] - g_m sum_{l kept} dlogg_l,   m < C_i
  (from ds_m = g_m (dg_m - sum_l g_l dg_l) with dg_l = 0 for dropped blocks).
  Outer gate position (Sec. 4.2 gate position, o = softmax(z) (g . V) with
  z unbiased and w_j = g of key j's block, 1 on the current block):
    dV_j += p_j w_j dO_i,  dz_j = p_j (w_j dp_j - Delta_i)  (Delta_i = dO_i . o_i),
    dlogg_m = sum_{j in B_m} p_j w_j dp_j   (= g_m dL/dg_m).
  Other gate activations of Sec. 4.2 (inner position): the gates are
  independent of one another, so only kept blocks get a score gradient,
  ds_m = dlogg_m d(log g_m)/ds_m: sigmoid, dlogg_m (1 - g_m); raw logit
  (log g = s), dlogg_m.

Selection (which blocks are kept) is taken from the forward: the gradient
treats it as fixed, as the kernels do.

GQA (sas_attention_bwd_gqa): a group's K, V and log-gates feed its G query
heads, so dK, dV and d(log g) are sums over the heads, and the score
gradient applies the gate softmax's Jacobian to the summed d(log g).

Full training scope (Sec. 4.2 "training scope", Eq. scope_grad): every
historical block is gated and nothing is dropped, which is the sparse form
with K >= C_i; its gradients are sas_attention_bwd_head with topk >= C
(sas_attention_bwd_full_head).

Hard Top-K gate with the straight-through estimator (Sec. 4.2 "ranking
preservation", App. D "hard gating with STE", Eq. rank_unbounded;
sas_attention_bwd_ste_head): the forward gate is g^hard (1 on the kept
blocks, 0 on the dropped ones: the inference form, logits unbiased, the
normaliser LSE_S over the attended keys S only); the backward takes
g^hat = stopgrad(g^hard - g) + g with the soft g = softmax(s), so
  dQ, dK, dV  are those of the hard forward (constant gates),
  dg_m        = sum_{j in B_m} p~_j (dp_j - Delta),  p~_j = exp(z_j - LSE_S),
                for EVERY historical block m (z_j = sm_scale q.k_j; for a
                dropped block p~ is the unbounded weight of Eq. rank_unbounded),
  ds_l        = g_l (dg_l - sum_m g_m dg_m)   (the softmax Jacobian).
"""
from __future__ import annotations

import math

import numpy as np

from oracle.sas_oracle import (GATE_INNER, GATE_LOGIT, GATE_SIGMOID, GATE_SOFTMAX, MODE_INFER_HARD,
                               MODE_TRAIN_SOFT, _row_keys_and_bias, historical_count, log_gates)


def sas_attention_bwd_head(Q, K, V, s, dO, b, topk, mode=MODE_TRAIN_SOFT, sm_scale=None, act=GATE_SOFTMAX,
                           pos=GATE_INNER):
    """Gradients of one head's SAS forward (gate activation `act`, gate
    position `pos`).

    Q, K, V, dO: [N, d]; s: [N, >=C-1] selector scores (row i reads s[i, :C_i]).
    Returns dict with dQ, dK, dV [N, d], dlogg [N, topk] (aligned with the
    forward's ascending kept list, 0 where padded), ds [N, C] (score gradient,
    0 past each row's history) and Delta [N].
    """
    N, d = Q.shape
    if sm_scale is None:
        sm_scale = 1.0 / math.sqrt(d)
    C = -(-N // b)
    dQ = np.zeros((N, d))
    dK = np.zeros((N, d))
    dV = np.zeros((N, V.shape[1]))
    dlogg = np.zeros((N, max(topk, 1)))
    ds = np.zeros((N, C))
    Delta = np.zeros(N)
    for i in range(N):
        keys, bias, weight, sel, _ = _row_keys_and_bias(i, s[i], b, topk, mode, act, pos)
        z = sm_scale * (K[keys] @ Q[i]) + bias
        ez = np.exp(z - z.max())
        p = ez / ez.sum()
        o = (p * weight) @ V[keys]
        dp = V[keys] @ dO[i]
        Delta[i] = dO[i] @ o
        dz = p * (weight * dp - Delta[i])
        dQ[i] = sm_scale * (dz @ K[keys])
        np.add.at(dK, keys, sm_scale * np.outer(dz, Q[i]))
        np.add.at(dV, keys, np.outer(p * weight, dO[i]))
        # d(log g) of a block: the row sum of dz (inner), of p w dp (outer)
        gsum = dz if pos == GATE_INNER else p * weight * dp
        if mode != MODE_TRAIN_SOFT:
            continue
        # kept blocks come first in `keys`, b tokens each, in ascending order
        c = historical_count(i, b)
        lg_all = log_gates(np.asarray(s[i][:c], dtype=np.float64), act)
        dl = np.zeros(c)
        for e, m in enumerate(sel):
            dl[m] = gsum[e * b:(e + 1) * b].sum()
            dlogg[i, e] = dl[m]
        if c:
            ds[i, :c] = _score_grad(dl, lg_all, act)
    return {"dQ": dQ, "dK": dK, "dV": dV, "dlogg": dlogg[:, :topk], "ds": ds, "Delta": Delta}


def _score_grad(dl, lg, act):
    """ds over a row's history from dlogg (0 on dropped blocks) and log g."""
    g = np.exp(lg)
    if act == GATE_SIGMOID:
        return dl * (1.0 - g)
    if act == GATE_LOGIT:
        return dl.copy()
    return dl - g * dl.sum()


def backward_flops_head(N, b, topk, d, sel_counts=None):
    """Algorithmic FLOPs of the backward of one head: per attended (row, key)
    pair the four products q.k, dO.v, dS k (into dQ) and the two key-side
    products dS^T q and P^T dO, 2 d FLOPs each -> 10 d per pair (Alg. 4 runs
    q.k and dO.v in both passes: the kernels execute 14 d)."""
    pairs = 0
    for i in range(N):
        c = i // b
        kept = min(topk, c)
        pairs += kept * b + (i - c * b + 1)
    return 10 * d * pairs


def sas_attention_bwd_gqa(Q, K, V, s, dO, b, topk, mode=MODE_TRAIN_SOFT, sm_scale=None, act=GATE_SOFTMAX,
                          pos=GATE_INNER):
    """Gradients of the GQA forward (group-shared selection, Sec. 5.3) of one
    batch element.  Q, dO: [Hq, N, d]; K, V: [Hkv, N, d]; s: [Hkv, N, >=C-1];
    Hq = G Hkv, query head h uses group h // G.  A group's K, V and log-gates
    enter the logits of all its G heads, so their gradients are the sums of
    the heads' contributions: dK_g, dV_g, dlogg_g = sum over the group of the
    per-head terms, and the score gradient applies the gate softmax's
    Jacobian (App. D) to the summed dlogg: ds_m = dl_m [m kept] - g_m sum dl.
    Returns dict with dQ [Hq, N, d], dK, dV [Hkv, N, d], dlogg [Hkv, N, topk],
    ds [Hkv, N, C].
    """
    Hq, N, d = Q.shape
    Hkv = K.shape[0]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    C = -(-N // b)
    dQ = np.zeros_like(Q, dtype=np.float64)
    dK = np.zeros((Hkv, N, d))
    dV = np.zeros((Hkv, N, V.shape[2]))
    dlogg = np.zeros((Hkv, N, max(topk, 1)))[:, :, :topk]
    ds = np.zeros((Hkv, N, C))
    for h in range(Hq):
        g = h // G
        r = sas_attention_bwd_head(Q[h], K[g], V[g], s[g], dO[h], b, topk, mode, sm_scale, act, pos)
        dQ[h] = r["dQ"]
        dK[g] += r["dK"]
        dV[g] += r["dV"]
        dlogg[g] += r["dlogg"]
    if mode == MODE_TRAIN_SOFT:
        for g in range(Hkv):
            for i in range(N):
                c = historical_count(i, b)
                if c == 0:
                    continue
                _, _, _, sel, _ = _row_keys_and_bias(i, s[g, i], b, topk, mode, act, pos)
                dl = np.zeros(c)
                for e, m in enumerate(sel):
                    dl[m] = dlogg[g, i, e]
                ds[g, i, :c] = _score_grad(dl, log_gates(np.asarray(s[g, i][:c], dtype=np.float64), act), act)
    return {"dQ": dQ, "dK": dK, "dV": dV, "dlogg": dlogg, "ds": ds}


def sas_attention_bwd_varlen(Q, K, V, s, dO, cu_seqlens, b, topk, mode=MODE_TRAIN_SOFT, sm_scale=None):
    """Gradients of the packed variable-length forward: every sequence
    (rows cu[k] .. cu[k+1]-1) is its own problem, so its gradients are those
    of the GQA backward on its slice, and nothing crosses sequences.
    Q, dO: [Hq, total, d]; K, V: [Hkv, total, d]; s: [Hkv, total, >=C-1]
    (C from the longest sequence).  Returns the fields of
    sas_attention_bwd_gqa on the whole token axis (ds has the columns of s
    that a sequence's rows can read; rows past cu[S] stay zero)."""
    Hq, total, d = Q.shape
    Hkv = K.shape[0]
    cu = [int(x) for x in cu_seqlens]
    Cs = s.shape[2]
    out = {"dQ": np.zeros((Hq, total, d)), "dK": np.zeros((Hkv, total, d)), "dV": np.zeros((Hkv, total, V.shape[2])),
           "dlogg": np.zeros((Hkv, total, topk)), "ds": np.zeros((Hkv, total, Cs))}
    for s0, s1 in zip(cu[:-1], cu[1:]):
        if s1 == s0:
            continue
        r = sas_attention_bwd_gqa(Q[:, s0:s1], K[:, s0:s1], V[:, s0:s1], s[:, s0:s1], dO[:, s0:s1], b, topk,
                                  mode, sm_scale)
        for f in ("dQ", "dK", "dV", "dlogg"):
            out[f][:, s0:s1] = r[f]
        out["ds"][:, s0:s1, :r["ds"].shape[2]] = r["ds"]
    return out


def sas_attention_bwd_full_head(Q, K, V, s, dO, b, sm_scale=None):
    """Gradients of the full training scope of one head (every historical
    block gated with log g = log_softmax(s) over the row's history): the
    sparse backward keeping every block.  dlogg is [N, C] indexed by block."""
    N = Q.shape[0]
    C = -(-N // b)
    return sas_attention_bwd_head(Q, K, V, s, dO, b, C, MODE_TRAIN_SOFT, sm_scale)


def sas_attention_bwd_ste_head(Q, K, V, s, dO, b, topk, sm_scale=None):
    """Gradients of the hard Top-K gate under the straight-through estimator,
    one head (see the module docstring).  Q, K, V, dO: [N, d]; s: [N, >=C-1].
    Returns dQ, dK, dV [N, d] (the hard forward's), dg [N, C] (dL/dg^hat of
    every historical block, 0 past the history), x = g dg [N, C] (the
    gradient with respect to log g^hat through the estimator) and ds [N, C]."""
    N, d = Q.shape
    if sm_scale is None:
        sm_scale = 1.0 / math.sqrt(d)
    C = -(-N // b)
    hard = sas_attention_bwd_head(Q, K, V, s, dO, b, topk, MODE_INFER_HARD, sm_scale)
    dg = np.zeros((N, C))
    x = np.zeros((N, C))
    ds = np.zeros((N, C))
    for i in range(N):
        c = historical_count(i, b)
        if c == 0:
            continue
        # the hard forward of row i: its attended keys, logits and normaliser
        keys, bias, _, _, _ = _row_keys_and_bias(i, s[i], b, topk, MODE_INFER_HARD)
        zs = sm_scale * (K[keys] @ Q[i]) + bias
        zmax = zs.max()
        lse_s = zmax + math.log(np.exp(zs - zmax).sum())
        o = np.exp(zs - lse_s) @ V[keys]
        delta = dO[i] @ o
        # every historical block, attended or not, under the same normaliser
        for m in range(c):
            toks = np.arange(m * b, (m + 1) * b)
            pt = np.exp(sm_scale * (K[toks] @ Q[i]) - lse_s)
            dg[i, m] = (pt * (V[toks] @ dO[i] - delta)).sum()
        g = np.exp(log_gates(np.asarray(s[i][:c], dtype=np.float64)))
        x[i, :c] = g * dg[i, :c]
        ds[i, :c] = g * (dg[i, :c] - (g * dg[i, :c]).sum())
    return {"dQ": hard["dQ"], "dK": hard["dK"], "dV": hard["dV"], "dg": dg, "x": x, "ds": ds}


def sas_attention_bwd_ste_gqa(Q, K, V, s, dO, b, topk, sm_scale=None):
    """The hard-STE gradients under GQA: Q, dO [Hq, N, d]; K, V, s per KV
    group.  dK, dV and the group's dg (hence x and ds) are sums over its G
    query heads; ds applies the Jacobian to the summed dg."""
    Hq, N, d = Q.shape
    Hkv = K.shape[0]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    C = -(-N // b)
    out = {"dQ": np.zeros((Hq, N, d)), "dK": np.zeros((Hkv, N, d)), "dV": np.zeros((Hkv, N, V.shape[2])),
           "dg": np.zeros((Hkv, N, C)), "x": np.zeros((Hkv, N, C)), "ds": np.zeros((Hkv, N, C))}
    for h in range(Hq):
        g = h // G
        r = sas_attention_bwd_ste_head(Q[h], K[g], V[g], s[g], dO[h], b, topk, sm_scale)
        out["dQ"][h] = r["dQ"]
        out["dK"][g] += r["dK"]
        out["dV"][g] += r["dV"]
        out["dg"][g] += r["dg"]
    for g in range(Hkv):
        for i in range(N):
            c = historical_count(i, b)
            if c == 0:
                continue
            gates = np.exp(log_gates(np.asarray(s[g, i][:c], dtype=np.float64)))
            dgi = out["dg"][g, i, :c]
            out["x"][g, i, :c] = gates * dgi
            out["ds"][g, i, :c] = gates * (dgi - (gates * dgi).sum())
    return out
