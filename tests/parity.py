"""Helpers shared by the GPU parity tests: run the C ABI on seeded inputs,
run the oracle on the same (bf16-rounded) inputs, compare.

Tolerances (written here once, used by every parity test):
  * indices (sel_idx, tile unions): bit-exact whenever the scores are given;
    with the learned selector, bit-exact on rows whose K-th / (K+1)-th score
    margin exceeds the bound on how far the GPU's fp32 score may sit from
    the oracle's (selector_score_bound), and a valid Top-K set on the rest.
  * O (bf16): max |err| <= 2e-2 and mean |err| <= 2e-3 against the fp64
    oracle, absolute, wherever O is a convex combination of value rows (every
    gate g <= 1: softmax and sigmoid activations, the inner position, the
    inference form, GQA, packed sequences, decode).  Two outputs are sums
    whose terms are not bounded by |v|, and get a derived extra term on top
    (outer_logit_extra, grad_extra): the outer position with the raw-logit
    activation (g = e^s > 1 scales probabilities after the softmax) and the
    backward's dQ, dK, dV (sums over many rows or keys).
  * LSE (fp32): max |err| <= 1e-2.
  * sel_logg (fp32, log g = s - LSE over up to ~1200 blocks): max |err| <= 1e-4.
"""
from __future__ import annotations

import math
import os

import numpy as np
import torch

from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth

O_MAX_ABS = 2e-2
O_MEAN_ABS = 2e-3
LSE_MAX_ABS = 1e-2
LOGG_MAX_ABS = 1e-4


def f64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def sample_rows(N, n_random=256, seed=0):
    """Rows 0..64, every block boundary +-1, the last 64 rows, and random rows."""
    rows = set(range(min(N, 65)))
    for m in range(64, N, 64):
        rows.update({m - 1, m, m + 1})
    rows.update(range(max(0, N - 64), N))
    rng = np.random.default_rng(seed)
    rows.update(rng.integers(0, N, size=min(n_random, N)).tolist())
    return np.array(sorted(r for r in rows if 0 <= r < N))


def run_gpu(B, H, N, d, topk, mode, Q, K, V, scores=None, Wq=None, Wk=None, d_sel=0,
            act=sas.SAS_GATE_SOFTMAX, pos=sas.SAS_GATE_INNER):
    sel = sas.SAS_SEL_SCORES_GIVEN if scores is not None else sas.SAS_SEL_MEANPOOL_PROJ
    layer = sas.SasLayer(B, H, N, d, topk, mode=mode, selector=sel, d_sel=d_sel, gate_act=act, gate_pos=pos)
    dev = torch.device("cuda:0")
    cu = lambda t: None if t is None else t.to(dev).contiguous()
    O, LSE, si, sl = layer.attention(cu(Q), cu(K), cu(V), cu(scores), cu(Wq), cu(Wk))
    T = -(-N // 128)
    unions = sas.sas_get_tile_union_counts(layer.h, B * H * T)
    status = sas.sas_get_device_status(layer.h)
    launches = sas.sas_launch_count(layer.h)
    layer.close()
    return {"O": O.cpu(), "LSE": LSE.cpu(), "sel_idx": si.cpu(), "sel_logg": sl.cpu(),
            "unions": np.array(unions).reshape(B, H, T), "status": status, "launches": launches}


def oracle_scores(Q, K, Wq, Wk, bi, hi):
    return OR.selector_scores(f64(Q[bi, hi]), f64(K[bi, hi]), f64(Wq[hi]), f64(Wk[hi]), 64)


# worst errors seen by compare_o, per test (printed in the terminal summary)
WORST = {}


def _record(what, mx, mean, derived):
    test = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]
    key = (test, what.split("[")[0] + (" (derived bound)" if derived else ""))
    old = WORST.get(key, (0.0, 0.0))
    WORST[key] = (max(old[0], mx), max(old[1], mean))


def compare_o(gpu_O, ref_O, what="O", extra=None):
    """Max and mean abs error of a bf16 output against the oracle.

    extra=None: the stated absolute bounds, max <= 2e-2, mean <= 2e-3.
    extra (same shape as ref_O): a derived per-element error bound of the
    output's own arithmetic, added to the stated bound element by element
    (max) and on average (mean); see outer_logit_extra and grad_extra."""
    err = np.abs(gpu_O - ref_O)
    if extra is None:
        mx, mean = float(err.max(initial=0.0)), float(err.mean()) if err.size else 0.0
        _record(what, mx, mean, False)
        assert mx <= O_MAX_ABS, f"{what}: max abs err {mx:.3e} > {O_MAX_ABS}"
        assert mean <= O_MEAN_ABS, f"{what}: mean abs err {mean:.3e} > {O_MEAN_ABS}"
        return mx, mean
    extra = np.broadcast_to(extra, err.shape)
    over = err - (O_MAX_ABS + extra)
    mx, mean = float(err.max(initial=0.0)), float(err.mean()) if err.size else 0.0
    _record(what, mx, mean, True)
    assert float(over.max(initial=-1.0)) <= 0, (
        f"{what}: max abs err {mx:.3e}, worst excess over 2e-2 + derived bound {float(over.max()):.3e}")
    mean_bound = O_MEAN_ABS + (float(extra.mean()) if extra.size else 0.0)
    assert mean <= mean_bound, f"{what}: mean abs err {mean:.3e} > {mean_bound:.3e}"
    return mx, mean


def outer_logit_extra(Q, K, V, s, b, topk, mode, rows, act, pos):
    """Derived extra bound for the outer position with the raw-logit gate.

    There O_i = sum_j p_j g_j v_j with g_j = e^{s} unbounded, so O is not a
    convex combination of value rows.  Each term p_j g_j is rounded to bf16
    before the PV product (relative error <= 2^-9) and O is rounded to bf16
    on output (<= 2^-9 |O_i| <= 2^-9 A_i), where A_i = sum_j p_j g_j |v_j| is
    the same sum over absolute values -- the oracle's output on |V|.  The
    extra term is 2^-8 A_i (first order; fp32 accumulation is far below)."""
    if not (act == OR.GATE_LOGIT and pos == OR.GATE_OUTER):
        return None
    A = OR.sas_attention_head(Q, K, np.abs(V), s, b, topk, mode, rows=rows, act=act, pos=pos)["O"]
    return 2.0 ** -8 * A


def grad_extra(Q, K, V, s, dO, O_gpu, b, topk, mode, sm_scale=None, act=OR.GATE_SOFTMAX, pos=OR.GATE_INNER):
    """Derived extra bounds for the backward's dQ, dK, dV of one head.

    dV_j = sum_i P_ij dO_i, dK_j = scale sum_i dS_ij q_i and dQ_i = scale sum_j
    dS_ij k_j are sums over up to thousands of terms, so their rounding error
    scales with the sums of absolute terms, not with |v|.  Per term the kernel
    rounds P and dS = P (dP - Delta) to bf16 (relative 2^-9), and Delta =
    dO.O uses the forward's bf16 O, which may sit dDelta_i = 2^-8 sum_c
    |dO_ic O_ic| from the exact value (moving dS_ij by P_ij dDelta_i); the
    output is rounded to bf16 (2^-9 of its value).  First order:
      E_S    = 2^-9 |dS| + P dDelta
      dQ: scale E_S |K| + 2^-9 |dQ|,   dK: scale E_S^T |Q| + 2^-9 |dK|,
      dV: 2^-9 P^T |dO| + 2^-9 |dV|,
    each doubled to cover the second-order and fp32 terms.  P comes from the
    oracle's materialised forward (Q, K, V [N, d]; s the head's scores).
    Outer gate position: P is the plain softmax and each key carries its
    block's gate w, so dV takes (P w)^T dO and dS = P (w dP - Delta)."""
    N, d = Q.shape
    if sm_scale is None:
        sm_scale = 1.0 / math.sqrt(d)
    mat = OR.sas_attention_materialized(Q, K, V, s, b, topk, mode, sm_scale, act=act, pos=pos)
    P, W = mat["P"], mat["gate"]
    dP = dO @ V.T
    Delta = (P * W * dP).sum(axis=1)
    dS = P * (W * dP - Delta[:, None])
    dDelta = 2.0 ** -8 * np.abs(dO * O_gpu).sum(axis=1)
    ES = 2.0 ** -9 * np.abs(dS) + P * dDelta[:, None]
    dQ = sm_scale * dS @ K
    dK = sm_scale * dS.T @ Q
    dV = (P * W).T @ dO
    return {"dQ": 2 * (sm_scale * ES @ np.abs(K) + 2.0 ** -9 * np.abs(dQ)),
            "dK": 2 * (sm_scale * ES.T @ np.abs(Q) + 2.0 ** -9 * np.abs(dK)),
            "dV": 2 * (2.0 ** -9 * (P * W).T @ np.abs(dO) + 2.0 ** -9 * np.abs(dV))}


def _flip_size(x, delta):
    """Size of a possible bf16 rounding disagreement for each value of x.

    The GPU rounds an fp32 value that may differ from the exact x by up to
    delta; the two roundings can only disagree when x lies within delta of a
    midpoint between two bf16 neighbours.  Where that can happen the
    disagreement is at most two bf16 steps of |x|; elsewhere it is zero.
    """
    b = OR.round_to_bf16(x)
    _, e = np.frexp(np.where(b == 0, 1.0, b))
    step = np.ldexp(1.0, np.maximum(e - 1, -126) - 7)
    dist_to_mid = step / 2 - np.abs(x - b)
    return np.where(dist_to_mid <= delta, 2 * step, 0.0)


def selector_score_bound(Q, K, Wq, Wk, bi, hi, d_sel, rows=None):
    """Per-row bound on |s_gpu - s_oracle| over the row's history, times two
    (the K-th and the (K+1)-th score may both move).  Returned for `rows`
    (default: all rows).

    The learned selector computes q~ = bf16(Wq q) and K~ = bf16(Wk mean(K_B))
    with fp32 accumulation (at most 128 terms, error <= 2^-17 of the sum of
    absolute products, doubled for the mean-pool sum), then s = q~.K~ / sqrt(d_sel)
    in fp32.  A coordinate contributes a possible bf16 disagreement only when
    its exact value sits within that accumulation error of a rounding midpoint.
    """
    q, k, wq, wk = f64(Q[bi, hi]), f64(K[bi, hi]), f64(Wq[hi]), f64(Wk[hi])
    rows = np.arange(q.shape[0]) if rows is None else np.asarray(rows)
    q = q[rows]
    qe = q @ wq.T
    dq = 2.0 ** -17 * (np.abs(q) @ np.abs(wq).T)
    kbar = OR.block_summaries(k, 64)
    ke = kbar @ wk.T
    dk = 2.0 ** -16 * (OR.block_summaries(np.abs(k), 64) @ np.abs(wk).T)
    fq, fk = _flip_size(qe, dq), _flip_size(ke, dk)
    qt, kt = np.abs(OR.round_to_bf16(qe)), np.abs(OR.round_to_bf16(ke))
    if kt.shape[0] == 0:
        return np.full(len(rows), 1e-30)
    bound = (fq @ kt.T + qt @ fk.T + fq @ fk.T + 2.0 ** -17 * (qt @ kt.T)) / np.sqrt(d_sel)
    bound += 2.0 ** -22 * np.abs(OR.round_to_bf16(qe) @ OR.round_to_bf16(ke).T) / np.sqrt(d_sel)
    tol = np.zeros(len(rows))
    for r, i in enumerate(rows):
        c = int(i) // 64
        if c > 0:
            tol[r] = 2 * bound[r, :c].max()
    return tol + 1e-30


def check_selection_rows(gpu_idx, s_rows, rows, topk, tol=None):
    """Checks every sampled row's kept set.

    With tol None (scores given) the set must equal the oracle's Top-K.
    Otherwise rows whose K-th/(K+1)-th margin exceeds tol[r] must match
    exactly and the others must hold a valid Top-K set within tol.
    Returns (exact_rows, near_tie_rows, mismatched_row_mask).
    """
    exact = near = 0
    mismatch = np.zeros(len(rows), dtype=bool)
    for r, i in enumerate(rows):
        c = i // 64
        hist = s_rows[r][:c]
        g = gpu_idx[r]
        nsel = min(topk, c)
        assert np.all(g[nsel:] == -1), f"row {i}: padding"
        gs = g[:nsel]
        assert np.all(np.diff(gs) > 0), f"row {i}: not strictly ascending"
        assert np.all((gs >= 0) & (gs < c)), f"row {i}: index out of range"
        ref = OR.topk_blocks(hist, topk)
        if tol is None:
            assert np.array_equal(gs, ref), f"row {i}: kept {gs} != oracle {ref}"
            exact += 1
            continue
        if c <= topk:
            assert np.array_equal(gs, ref)
            exact += 1
            continue
        srt = np.sort(hist)[::-1]
        margin = srt[topk - 1] - srt[topk]
        if margin > tol[r]:
            if not np.array_equal(gs, ref):
                raise AssertionError(f"row {i}: kept {gs} != oracle {ref} with margin {margin:.3e} > tol {tol[r]:.3e}")
            exact += 1
        else:
            near += 1
            assert hist[gs].min() >= srt[topk - 1] - tol[r], f"row {i}: kept block far below the K-th score"
            mismatch[r] = not np.array_equal(gs, ref)
    return exact, near, mismatch


def oracle_union_counts(sel_idx_full, N, topk):
    """Per 128-row tile: number of distinct kept blocks below the tile's diagonal (2t)."""
    T = -(-N // 128)
    out = np.zeros(T, dtype=np.int64)
    for t in range(T):
        rows = sel_idx_full[t * 128:min(N, (t + 1) * 128)]
        v = rows[rows >= 0]
        out[t] = len(set(v[v < 2 * t].tolist()))
    return out
