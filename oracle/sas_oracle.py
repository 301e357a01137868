"""Plain fp64 CPU oracle for the SAS attention forward and the dense GELU MLP.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: only the tests, the smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the CUDA library; the two meet
only through the seeded input generator, which holds none of the method's
arithmetic.

What it computes (SAS, "Simple Attention Sparsification", arXiv 2609.13141):

  a1  block summaries      Kbar_m = mean of the keys of block B_m            (App. B, Limitation: pooled block summaries)
  a2  selector scores      s_im = R_theta(q_i, {K_Bm})                       (Alg. 1 step 1; Sec. 4.3)
  a3  causal log-gates     log g_m = s_m - LSE(s) over the row's history     (Eq. normalized_log_gate)
  a4  Top-K selection      I = TopK(g, K) = TopK(s, K)                       (Eq. selected_context; Alg. 1 / Alg. 2)
  a5  gated attention      o = softmax(q K_S^T + log g_S) V_S                (Eq. ours_train; Alg. 2 for the ungated form)
      ablation forms       gate activation softmax / sigmoid / logit and gate position inner / outer
                           (Sec. 4.2, Components of learnable ranking; Eq. general_gate)
      training scopes      full scope: every historical block gated, no Top-K (Table 1 setting 9);
                           full*: noise added to s before activation and Top-K (Table 1 setting 11)
  a6  dense MLP (not SAS)  Y = GELU(X W1^T + b1) W2^T + b2, exact-erf GELU

Readings of points the paper leaves open (each one is also listed with its
reasoning in the design notes of the repository):

  * sm_scale multiplies q.k only; the log-gate is added unscaled (Alg. 3,
    gated_scores).
  * Token j is in block floor(j / b).  For query i the current block B_0 is
    block floor(i / b), restricted causally to keys j <= i, always kept with a
    unit gate; its historical blocks are 0 .. floor(i / b) - 1, so
    C_i = floor(i / b) (Sec. 4.1, Eq. general_gate).
  * The gate softmax runs over all C_i historical blocks of the row, not only
    the selected ones, and is not renormalised after selection (Eq.
    normalized_log_gate; Eq. scope_grad).
  * Top-K is exact-K: order by (score descending, block index ascending), so a
    tie goes to the lower block index.  Rows with C_i <= K keep every
    historical block; K = 0 keeps none (only the current block).
  * Selection uses the scores s, never the computed log-gates (the two orders
    agree because log g = s - const; Alg. 1 vs Alg. 2).
  * Selector R_theta (MEANPOOL_PROJ): the paper names the AttnGate of
    SeerAttention-R without describing it.  The reading used here is
    q~_i = bf16(Wq q_i), K~_m = bf16(Wk Kbar_m), s_im = q~_i . K~_m / sqrt(d_s),
    with Wq, Wk in linear-layer layout [d_s, d].  The two projections are
    bf16 activations, as in a bf16 model.
    PARITY UNPINNED for the selector architecture itself: no paper value
    exists to check it against; only its arithmetic is pinned.
  * MLP: the hidden activation GELU(X W1^T + b1) is a bf16 tensor between the
    two products (the precision of a stored bf16 activation).
  * GQA: the G query heads of a KV group share one selection (Sec. 5.3); with
    the learned selector the group's gate query is q~ = bf16(Wq_g [q_0; ...;
    q_{G-1}]), Wq_g [d_s, G d] (the paper does not say how the heads combine).
  * Packed sequences: each is its own causal problem; its blocks start at its
    first token.

Arrays are float64 numpy arrays holding the bf16-rounded inputs the GPU sees.
One "head" means one (batch, head) pair; Q, K, V of a head are [N, d].
"""
from __future__ import annotations

import math

import numpy as np

MODE_TRAIN_SOFT = 0   # Eq. ours_train: selected historical blocks get + log g
MODE_INFER_HARD = 1   # Alg. 2: selected historical blocks get no bias

# Gate activation phi of Eq. general_gate (Sec. 4.2, gate activation):
GATE_SOFTMAX = 0      # g = softmax(s) over the row's historical blocks (the SAS default)
GATE_SIGMOID = 1      # g = sigmoid(s), independent gates
GATE_LOGIT = 2        # s added to the logits directly, i.e. log g = s
# Gate position (Sec. 4.2, gate position):
GATE_INNER = 0        # o = softmax(q K^T + log g) V  (the SAS default)
GATE_OUTER = 1        # o = softmax(q K^T) (g . V): gates scale the value rows after the softmax


# ---------------------------------------------------------------- rounding --

def round_to_bf16(x):
    """Round float64 values to the nearest bfloat16 value, ties to even.

    bfloat16 keeps 8 significant bits and the float32 exponent range.  For a
    value with binary exponent e (2**e <= |x| < 2**(e+1)) the spacing of
    bfloat16 numbers is 2**(e-7); below 2**-126 the spacing stays 2**-133
    (subnormals).  Division by a power of two is exact, and numpy's rint
    rounds half to even, so this is a single correctly rounded step.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros_like(x)
    nz = x != 0
    _, e = np.frexp(x[nz])               # x = m * 2**e with 0.5 <= |m| < 1
    e = np.maximum(e - 1, -126)          # floor(log2|x|), clamped at the subnormal range
    ulp = np.ldexp(1.0, e - 7)
    out[nz] = np.rint(x[nz] / ulp) * ulp
    return out


# ----------------------------------------------------------- block layout --

def num_blocks(N, b):
    """C = ceil(N / b) contiguous token blocks (Sec. 3, block partition)."""
    return -(-N // b)


def historical_count(i, b):
    """C_i = floor(i / b): blocks strictly before query i's current block (Sec. 4.1)."""
    return i // b


# --------------------------------------------------------------- a1 / a2 --

def block_summaries(K, b):
    """a1: Kbar[m] = (1/b) * sum of k_j over the b tokens j of block m.

    Only full blocks are summarised (m < floor(N / b)): a partial last block
    is never historical for any query, because a query's historical blocks all
    precede its own block.
    """
    N, d = K.shape
    F = N // b
    out = np.zeros((F, d))
    for m in range(F):
        out[m] = K[m * b:(m + 1) * b].sum(axis=0) / b
    return out


def selector_scores(Q, K, Wq, Wk, b):
    """a2 (MEANPOOL_PROJ reading of R_theta): s[i, m] for every row i, m < F.

    q~_i = bf16(Wq q_i), K~_m = bf16(Wk Kbar_m), s_im = q~_i . K~_m / sqrt(d_s).
    Entries with m >= C_i are computed but never used by a row (causality).
    Wq, Wk: [d_s, d] (linear-layer layout [out, in]).
    """
    d_s = Wq.shape[0]
    qt = round_to_bf16(Q @ Wq.T)
    kt = round_to_bf16(block_summaries(K, b) @ Wk.T)
    return (qt @ kt.T) / math.sqrt(d_s)


def selector_scores_group(Qg, K, Wq_g, Wk, b):
    """a2 for a GQA group (MEANPOOL_PROJ reading, group gate query): one score
    table for the G query heads of a KV group, so that they share one Top-K
    (Sec. 5.3).  The paper does not say how the G heads form one gate query;
    the reading is q~_i = bf16(Wq_g [q_{0,i}; ...; q_{G-1,i}]) with
    Wq_g [d_s, G d] (G = 1 is selector_scores; averaging the heads is the
    special case Wq_g = [W ... W] / G), and K~_m = bf16(Wk Kbar_m) of the
    group's keys.  Qg: [G, N, d]; K: [N, d]; Wk: [d_s, d].
    """
    G, N, d = Qg.shape
    d_s = Wq_g.shape[0]
    qcat = np.concatenate([Qg[h] for h in range(G)], axis=1)   # [N, G d], head-major
    qt = round_to_bf16(qcat @ Wq_g.T)
    kt = round_to_bf16(block_summaries(K, b) @ Wk.T)
    return (qt @ kt.T) / math.sqrt(d_s)


# --------------------------------------------------------------- a3 / a4 --

def log_gates(s_hist, act=GATE_SOFTMAX):
    """a3, log g_m for the row's historical blocks.

    GATE_SOFTMAX: Eq. normalized_log_gate, log g_m = s_m - LSE(s) over the row's history.
    GATE_SIGMOID: g_m = sigmoid(s_m), so log g_m = -log(1 + exp(-s_m)).
    GATE_LOGIT:   s_m is injected into the logits unnormalised, log g_m = s_m.
    (Sec. 4.2, gate activation.)"""
    s_hist = np.asarray(s_hist, dtype=np.float64)
    if s_hist.size == 0:
        return s_hist.copy()
    if act == GATE_SIGMOID:
        return -np.logaddexp(0.0, -s_hist)
    if act == GATE_LOGIT:
        return s_hist.copy()
    mx = s_hist.max()
    lse = mx + math.log(np.exp(s_hist - mx).sum())
    return s_hist - lse


def topk_blocks(s_hist, K):
    """a4, Eq. selected_context: the K highest-scoring historical blocks.

    Exact-K with ties to the lower block index; all blocks when C_i <= K.
    Returned in ascending block order.
    """
    s_hist = np.asarray(s_hist)
    C_i = s_hist.shape[0]
    if C_i <= K:
        return np.arange(C_i)
    # A stable sort on the negated scores keeps equal scores in ascending
    # block order, which is the tie rule.
    order = np.argsort(-s_hist, kind="stable")
    return np.sort(order[:K])


# -------------------------------------------------------------------- a5 --

def _row_keys_and_bias(i, s_row, b, topk, mode, act=GATE_SOFTMAX, pos=GATE_INNER):
    """Attended keys of row i, their additive logit bias and their
    multiplicative weight on the probabilities.

    Inner position (Eq. ours_train): bias log g on the selected historical
    blocks, weight 1.  Outer position: bias 0, weight g (the gate scales the
    value rows after the softmax).  Inference mode (Alg. 2): neither.  The
    current block always has bias 0 and weight 1 (g_0 = 1, Eq. general_gate).

    Returns (keys, bias, weight, sel_idx, sel_logg) where keys lists token
    indices: first the tokens of the selected historical blocks, then the
    causal part of the current block.
    """
    c = historical_count(i, b)
    s_hist = np.asarray(s_row[:c], dtype=np.float64)
    lg = log_gates(s_hist, act)
    sel = topk_blocks(s_hist, topk)
    keys, bias, weight = [], [], []
    for m in sel:
        toks = np.arange(m * b, (m + 1) * b)
        keys.append(toks)
        gated = mode == MODE_TRAIN_SOFT
        bias.append(np.full(b, lg[m] if gated and pos == GATE_INNER else 0.0))
        weight.append(np.full(b, math.exp(lg[m]) if gated and pos == GATE_OUTER else 1.0))
    cur = np.arange(c * b, i + 1)           # current block, causal, unit gate
    keys.append(cur)
    bias.append(np.zeros(cur.shape[0]))
    weight.append(np.ones(cur.shape[0]))
    return np.concatenate(keys), np.concatenate(bias), np.concatenate(weight), sel, lg[sel]


def sas_attention_head(Q, K, V, s, b, topk, mode=MODE_TRAIN_SOFT, sm_scale=None,
                       rows=None, act=GATE_SOFTMAX, pos=GATE_INNER):
    """a5 for one head: O_i = sum_j softmax(z)_j w_j v_j, z_j = sm_scale q_i.k_j + bias_j
    (w_j = 1 except for the outer gate position, where w_j = g of key j's block).

    s: [N, >=C-1] selector scores of the head (row i reads s[i, :C_i]).
    rows: iterable of query indices (default: all).
    Returns dict with O [R, d], LSE [R], sel_idx [R, topk] (ascending, -1
    padded) and sel_logg [R, topk] (log g of the selected blocks, 0 padded).
    LSE is the natural-log log-sum-exp of the logits z (Alg. 3 output).
    """
    N, d = Q.shape
    if sm_scale is None:
        sm_scale = 1.0 / math.sqrt(d)
    rows = np.arange(N) if rows is None else np.asarray(rows)
    R = rows.shape[0]
    O = np.zeros((R, V.shape[1]))
    LSE = np.zeros(R)
    sel_idx = np.full((R, topk), -1, dtype=np.int64)
    sel_logg = np.zeros((R, topk))
    for r, i in enumerate(rows):
        keys, bias, weight, sel, lg = _row_keys_and_bias(int(i), s[i], b, topk, mode, act, pos)
        z = sm_scale * (K[keys] @ Q[i]) + bias
        zmax = z.max()
        w = np.exp(z - zmax)
        l = w.sum()
        O[r] = ((w * weight) @ V[keys]) / l
        LSE[r] = zmax + math.log(l)
        sel_idx[r, :sel.shape[0]] = sel
        sel_logg[r, :sel.shape[0]] = lg
    return {"O": O, "LSE": LSE, "sel_idx": sel_idx, "sel_logg": sel_logg}


def sas_attention_materialized(Q, K, V, s, b, topk, mode=MODE_TRAIN_SOFT,
                               sm_scale=None, act=GATE_SOFTMAX, pos=GATE_INNER):
    """Brute force: the whole N x N gated logit matrix, then a row softmax.

    This is the naive form the paper calls prohibitive (Sec. 4.3, Kernel
    Design); it exists only to cross-check the per-row oracle on small N.
    Bias[i, j] = 0 on the causal current block, log g (or 0 in inference
    mode) on selected historical blocks, -inf elsewhere.
    """
    N, d = Q.shape
    if sm_scale is None:
        sm_scale = 1.0 / math.sqrt(d)
    bias = np.full((N, N), -np.inf)
    gate = np.ones((N, N))
    for i in range(N):
        c = historical_count(i, b)
        s_hist = np.asarray(s[i][:c], dtype=np.float64)
        lg = log_gates(s_hist, act)
        for m in topk_blocks(s_hist, topk):
            gated = mode == MODE_TRAIN_SOFT
            bias[i, m * b:(m + 1) * b] = lg[m] if gated and pos == GATE_INNER else 0.0
            if gated and pos == GATE_OUTER:
                gate[i, m * b:(m + 1) * b] = math.exp(lg[m])
        bias[i, c * b:i + 1] = 0.0
    Z = sm_scale * (Q @ K.T) + bias
    zmax = Z.max(axis=1, keepdims=True)
    W = np.exp(Z - zmax)
    l = W.sum(axis=1, keepdims=True)
    return {"O": (W * gate @ V) / l, "LSE": (zmax + np.log(l))[:, 0], "P": W / l, "gate": gate}


def sas_attention(Q, K, V, b, topk, mode=MODE_TRAIN_SOFT, sm_scale=None,
                  scores=None, Wq=None, Wk=None, heads=None, rows=None,
                  act=GATE_SOFTMAX, pos=GATE_INNER):
    """Alg. 1 steps 1-4 (training forward) over [B, H, N, d] inputs.

    Either `scores` [B, H, N, >=C-1] are given (scores-given selector) or the
    MEANPOOL_PROJ selector weights Wq, Wk [H, d_s, d] are.  heads: list of
    (batch, head) pairs to evaluate (default all); rows as in
    sas_attention_head.  Returns {(bi, hi): result-dict}.
    """
    Bn, H, N, d = Q.shape
    heads = [(bi, hi) for bi in range(Bn) for hi in range(H)] if heads is None else heads
    out = {}
    for bi, hi in heads:
        if scores is not None:
            s = scores[bi, hi]
        else:
            s = selector_scores(Q[bi, hi], K[bi, hi], Wq[hi], Wk[hi], b)
        out[(bi, hi)] = sas_attention_head(Q[bi, hi], K[bi, hi], V[bi, hi], s, b,
                                           topk, mode, sm_scale, rows, act, pos)
    return out


def sas_attention_gqa(Q, K, V, b, topk, scores=None, mode=MODE_TRAIN_SOFT, sm_scale=None,
                      heads=None, rows=None, act=GATE_SOFTMAX, pos=GATE_INNER, Wq=None, Wk=None):
    """GQA form with group-shared selection (Sec. 5.3: the query heads of a
    GQA group share one Top-K; Sec. 5 inference implementation: Top-K per
    query group).  Q [B, Hq, N, d]; K, V [B, Hkv, N, d]; scores
    [B, Hkv, N, >=C-1], one table per KV group; Hq = G Hkv, query head h
    belongs to group h // G.  Every query head attends with its group's K,
    V, kept blocks and log-gates.  Without scores, the learned selector with
    the group gate query (selector_scores_group; Wq [Hkv, d_s, G d], Wk
    [Hkv, d_s, d]) gives each group's table.  Returns {(bi, h): result-dict}.
    """
    Bn, Hq, N, d = Q.shape
    Hkv = K.shape[1]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    heads = [(bi, hi) for bi in range(Bn) for hi in range(Hq)] if heads is None else heads
    out = {}
    tables = {}
    for bi, hi in heads:
        g = hi // G
        if scores is not None:
            sg = scores[bi, g]
        else:
            if (bi, g) not in tables:
                tables[(bi, g)] = selector_scores_group(Q[bi, g * G:(g + 1) * G], K[bi, g], Wq[g], Wk[g], b)
            sg = tables[(bi, g)]
        out[(bi, hi)] = sas_attention_head(Q[bi, hi], K[bi, g], V[bi, g], sg, b,
                                           topk, mode, sm_scale, rows, act, pos)
    return out


def sas_attention_varlen(Q, K, V, cu_seqlens, b, topk, scores=None, mode=MODE_TRAIN_SOFT, sm_scale=None,
                         act=GATE_SOFTMAX, pos=GATE_INNER, Wq=None, Wk=None):
    """Packed variable-length form: sequences s = 0 .. S-1 occupy rows
    cu_seqlens[s] .. cu_seqlens[s+1]-1 of the token axis; each is its own
    causal problem whose block partition starts at its first token (token t
    of sequence s is in its block floor(t / b); nothing crosses sequences).
    Q [Hq, total, d]; K, V [Hkv, total, d]; scores [Hkv, total, >=C-1], row
    cu[s] + t reading entries 0 .. floor(t / b) - 1; Hq = G Hkv (GQA, query
    head h uses group h // G).  Without scores, the learned selector with the
    group gate query (selector_scores_group; Wq [Hkv, d_s, G d], Wk
    [Hkv, d_s, d]) scores each sequence against the summaries of its own
    blocks.  Returns dict of [Hq, total, ...] O, LSE and [Hkv, total, topk]
    sel_idx / sel_logg (rows past cu[S] stay zero / -1).
    """
    Hq, total, d = Q.shape
    Hkv = K.shape[0]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    cu = [int(x) for x in cu_seqlens]
    if cu[0] != 0 or any(cu[k + 1] < cu[k] for k in range(len(cu) - 1)) or cu[-1] > total:
        raise ValueError("cu_seqlens must start at 0, not decrease and stay within the token axis")
    O = np.zeros((Hq, total, V.shape[2]))
    LSE = np.zeros((Hq, total))
    sel_idx = np.full((Hkv, total, topk), -1, dtype=np.int64)
    sel_logg = np.zeros((Hkv, total, topk))
    for s0, s1 in zip(cu[:-1], cu[1:]):
        if s1 == s0:
            continue
        tables = {}
        for h in range(Hq):
            g = h // G
            if scores is not None:
                sg = scores[g, s0:s1]
            else:
                if g not in tables:
                    tables[g] = selector_scores_group(Q[g * G:(g + 1) * G, s0:s1], K[g, s0:s1], Wq[g], Wk[g], b)
                sg = tables[g]
            r = sas_attention_head(Q[h, s0:s1], K[g, s0:s1], V[g, s0:s1], sg, b, topk, mode,
                                   sm_scale, None, act, pos)
            O[h, s0:s1] = r["O"]
            LSE[h, s0:s1] = r["LSE"]
            if h % G == 0:
                sel_idx[g, s0:s1] = r["sel_idx"]
                sel_logg[g, s0:s1] = r["sel_logg"]
    return {"O": O, "LSE": LSE, "sel_idx": sel_idx, "sel_logg": sel_logg}


# ------------------------------------------------------ training scopes --

def sas_attention_full_scope(Q, K, V, s, b, sm_scale=None, rows=None):
    """Full training scope (Table 1 setting 9: Eq. fula with the log-gates of
    Eq. ours_train; Sec. 4.2 "training scope"): no Top-K.  Row i attends to
    every key of its history; a key of historical block m < C_i gets the bias
    log g_m = s_m - LSE(s_0 .. s_{C_i - 1}) (Eq. normalized_log_gate), a key of
    the current block (j <= i) gets 0 (unit gate).
    Q, K, V [N, d]; s [N, >=C-1].  Returns dict with O [R, d] and LSE [R].
    """
    N, d = Q.shape
    if sm_scale is None:
        sm_scale = 1.0 / math.sqrt(d)
    rows = np.arange(N) if rows is None else np.asarray(rows)
    O = np.zeros((len(rows), V.shape[1]))
    LSE = np.zeros(len(rows))
    for r, i in enumerate(rows):
        i = int(i)
        c = historical_count(i, b)
        bias = np.zeros(i + 1)
        if c:
            hist = np.asarray(s[i][:c], dtype=np.float64)
            top = hist.max()
            lse = top + math.log(np.exp(hist - top).sum())
            bias[:c * b] = np.repeat(hist - lse, b)
        z = sm_scale * (K[:i + 1] @ Q[i]) + bias
        zmax = z.max()
        w = np.exp(z - zmax)
        O[r] = (w @ V[:i + 1]) / w.sum()
        LSE[r] = zmax + math.log(w.sum())
    return {"O": O, "LSE": LSE}


def noisy_scores(s, noise):
    """full* (Table 1 setting 11): noise is added to the selector scores before
    the gate activation, so both the Top-K choice and the gates use
    s~ = s + eps (Sec. 4.2: a stochastic approximation of the full scope).
    Reading: scores and noise are fp32 tensors and their sum is formed in fp32."""
    return (np.asarray(s, dtype=np.float32) + np.asarray(noise, dtype=np.float32)).astype(np.float64)


# -------------------------------------------------------------------- a6 --

def gelu(x):
    """Exact GELU: x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    x = np.asarray(x, dtype=np.float64)
    erf = np.vectorize(math.erf, otypes=[np.float64])
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def gelu_mlp(X, W1, W2, b1=None, b2=None, rows=None):
    """a6 (dense MLP; SAS does not define one): Y = bf16(GELU(X W1^T + b1)) W2^T + b2.

    X [T, D], W1 [F, D], W2 [D, F] (linear-layer weight layout [out, in]).
    rows: optional subset of token rows.
    """
    Xr = X if rows is None else X[np.asarray(rows)]
    Hh = Xr @ W1.T
    if b1 is not None:
        Hh = Hh + b1
    G = round_to_bf16(gelu(Hh))
    Y = G @ W2.T
    if b2 is not None:
        Y = Y + b2
    return Y


# ------------------------------------------------------------- accounting --

def attention_flops_row(i, b, topk, d, d_sel=0):
    """Algorithmic FLOPs of one query row: 4 d (|current| + b min(K, C_i)) + 2 d_s C_i."""
    c = historical_count(i, b)
    cur = i - c * b + 1
    return 4 * d * (cur + b * min(topk, c)) + 2 * d_sel * c
