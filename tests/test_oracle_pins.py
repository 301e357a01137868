"""Pins for the CPU oracle: each test checks the oracle against something
other than itself -- hand-derived closed forms (tests/golden), library
routines that implement a special case independently (torch SDPA, torch's
bf16 conversion, torch GELU, scipy logsumexp), invariants the paper states,
and brute force on tiny inputs.
"""
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

from oracle import sas_oracle as O
from paper_2609_13141_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "sas_worked_examples.json")


def f64(t):
    return t.to(torch.float64).numpy()


# ------------------------------------------------------------- bf16 rounding

def test_round_to_bf16_matches_torch_conversion():
    # float32 inputs have one rounding to bf16 in torch; the oracle rounds the
    # exact float64 value of the same float32 number, so both must agree bit for bit.
    x = synth.normal((20000,), seed=5, std=3.0)
    x = torch.cat([x, x * 1e-30, x * 1e30, torch.tensor([0.0, -0.0, 1.0, -2.5])])
    # exact ties between two bf16 neighbours: 1 + 2^-8 (tie, even -> 1), 1 + 3*2^-8 (tie -> up)
    x = torch.cat([x, torch.tensor([1 + 2.0**-8, 1 + 3 * 2.0**-8, -(1 + 2.0**-8), 2.0**-130 * 1.5])])
    ref = x.to(torch.bfloat16).to(torch.float64).numpy()
    got = O.round_to_bf16(x.to(torch.float64).numpy())
    assert np.array_equal(ref, got)


# ---------------------------------------------------------- a1 block summary

def test_block_summaries_closed_form_ramp_and_partial_block():
    b, N, d = 8, 8 * 5 + 3, 3
    j = np.arange(N, dtype=np.float64)
    K = np.stack([j, 2 * j, np.ones(N)], axis=1)
    Kbar = O.block_summaries(K, b)
    assert Kbar.shape == (5, d)            # the 3-token tail block is not summarised
    m = np.arange(5)
    mean_j = m * b + (b - 1) / 2.0         # mean of an arithmetic run
    assert np.allclose(Kbar[:, 0], mean_j)
    assert np.allclose(Kbar[:, 1], 2 * mean_j)
    assert np.allclose(Kbar[:, 2], 1.0)


def test_selector_worked_example():
    g = json.load(open(GOLDEN))["selector_example"]
    K = np.array(g["K"], float)
    Q = np.array(g["Q"], float)
    I2 = np.eye(2)
    assert np.allclose(O.block_summaries(K, g["b"]), g["expect_Kbar"])
    s = O.selector_scores(Q, K, I2, I2, g["b"])
    assert np.allclose(s[3], g["expect_s_row3"], rtol=0, atol=1e-15)


def test_selector_hand_example_projected():
    # Non-identity projections with d_s = 2 != d = 3 and Wq != Wk, values whose
    # projections fall between bf16 neighbours (one exactly on a midpoint):
    # the expected numbers are worked out by hand in the fixture.  A transposed
    # weight, a dropped bf16 rounding of q~ or K~, or sqrt(d) for sqrt(d_s)
    # each changes at least one of them.
    g = json.load(open(GOLDEN))["selector_example_projected"]
    K, Q = np.array(g["K"], float), np.array(g["Q"], float)
    Wq, Wk = np.array(g["Wq"], float), np.array(g["Wk"], float)
    assert np.array_equal(O.round_to_bf16(np.concatenate([K.ravel(), Q.ravel(), Wq.ravel(), Wk.ravel()])),
                          np.concatenate([K.ravel(), Q.ravel(), Wq.ravel(), Wk.ravel()]))
    assert np.array_equal(O.block_summaries(K, g["b"]), np.array(g["expect_Kbar"]))
    assert np.array_equal(O.round_to_bf16(Q[5] @ Wq.T), np.array(g["expect_qt_row5"]))
    assert np.array_equal(O.round_to_bf16(O.block_summaries(K, g["b"]) @ Wk.T), np.array(g["expect_Kt"]))
    s = O.selector_scores(Q, K, Wq, Wk, g["b"])
    assert s.shape == (6, 3)
    assert np.allclose(s[5, :2] * math.sqrt(2.0), g["expect_s_row5_times_sqrt2"], rtol=0, atol=1e-14)
    # the group form with G = 1 is the same selector
    sg = O.selector_scores_group(Q[None], K, Wq, Wk, g["b"])
    assert np.array_equal(sg, s)


def test_selector_scores_scaling_and_permutation():
    # doubling Wq (exact in bf16) doubles every score; permuting key blocks
    # permutes the score columns.
    rng = np.random.default_rng(0)
    b, N, d, ds = 4, 32, 8, 6
    Q = O.round_to_bf16(rng.standard_normal((N, d)))
    K = O.round_to_bf16(rng.standard_normal((N, d)))
    Wq = O.round_to_bf16(rng.standard_normal((ds, d)) * 0.3)
    Wk = O.round_to_bf16(rng.standard_normal((ds, d)) * 0.3)
    s = O.selector_scores(Q, K, Wq, Wk, b)
    assert np.allclose(O.selector_scores(Q, K, 2 * Wq, Wk, b), 2 * s, rtol=1e-12, atol=0)
    perm = rng.permutation(N // b)
    Kp = K.reshape(N // b, b, d)[perm].reshape(N, d)
    assert np.allclose(O.selector_scores(Q, Kp, Wq, Wk, b), s[:, perm], rtol=1e-12, atol=1e-15)


# ------------------------------------------------------------------ a3 gates

def test_log_gates_normalised_shift_invariant_and_single_block():
    rng = np.random.default_rng(1)
    for C in [1, 2, 7, 100]:
        s = rng.standard_normal(C) * 3
        lg = O.log_gates(s)
        assert math.isclose(np.exp(lg).sum(), 1.0, rel_tol=1e-12)      # softmax gates sum to 1
        assert np.allclose(O.log_gates(s + 17.25), lg, atol=1e-12)      # Eq. normalized_log_gate shift invariance
        assert np.allclose(lg, s - scipy.special.logsumexp(s), atol=1e-12)
    assert O.log_gates(np.array([4.2]))[0] == 0.0                      # one block: g = 1
    lg = O.log_gates(np.array([0.0, math.log(3.0)]))
    assert np.allclose(lg, [math.log(0.25), math.log(0.75)], atol=1e-15)


# ------------------------------------------------------------------ a4 top-K

def test_topk_brute_force_with_ties():
    rng = np.random.default_rng(2)
    for _ in range(300):
        C = int(rng.integers(0, 40))
        K = int(rng.integers(0, 12))
        s = rng.integers(0, 4, size=C).astype(np.float64)       # many exact ties
        got = list(O.topk_blocks(s, K))
        ranked = sorted(range(C), key=lambda m: (-s[m], m))       # score desc, index asc
        assert got == sorted(ranked[:K])


def test_topk_all_when_history_short_and_none_when_k0():
    s = np.array([0.3, -1.0, 2.0])
    assert list(O.topk_blocks(s, 3)) == [0, 1, 2]
    assert list(O.topk_blocks(s, 10)) == [0, 1, 2]
    assert list(O.topk_blocks(s, 0)) == []
    assert list(O.topk_blocks(s, 1)) == [2]


# ------------------------------------------------------------ a5 attention

@pytest.mark.parametrize("case", json.load(open(GOLDEN))["cases"], ids=lambda c: c["name"])
def test_attention_worked_examples(case):
    Q = np.array(case["Q"], float)
    K = np.array(case["K"], float)
    V = np.array(case["V"], float)
    N = Q.shape[0]
    s = np.zeros((N, N))
    s[case["row"], :len(case["scores_row"])] = case["scores_row"]
    mode = O.MODE_TRAIN_SOFT if case["mode"] == "train" else O.MODE_INFER_HARD
    r = O.sas_attention_head(Q, K, V, s, case["b"], case["topk"], mode,
                             case["sm_scale"], rows=[case["row"]])
    nsel = len(case["expect_sel_idx"])
    assert list(r["sel_idx"][0, :nsel]) == case["expect_sel_idx"]
    assert np.all(r["sel_idx"][0, nsel:] == -1)
    assert np.allclose(r["sel_logg"][0, :nsel], case["expect_sel_logg"], atol=1e-14)
    assert np.allclose(r["O"][0], case["expect_O"], atol=1e-14)
    assert math.isclose(r["LSE"][0], case["expect_LSE"], abs_tol=1e-14)


def _rand_head(N, d, seed):
    rng = np.random.default_rng(seed)
    q = O.round_to_bf16(rng.standard_normal((N, d)))
    k = O.round_to_bf16(rng.standard_normal((N, d)))
    v = O.round_to_bf16(rng.standard_normal((N, d)))
    return q, k, v, rng


def _sdpa(q, k, v, mask, scale):
    t = lambda a: torch.from_numpy(a)[None, None]
    return F.scaled_dot_product_attention(t(q), t(k), t(v), attn_mask=t(mask), scale=scale)[0, 0].numpy()


@pytest.mark.parametrize("N,b", [(37, 8), (64, 16), (5, 8)])
def test_infer_keep_all_equals_dense_causal_sdpa(N, b):
    q, k, v, rng = _rand_head(N, 16, 3)
    s = rng.standard_normal((N, N))
    C = O.num_blocks(N, b)
    r = O.sas_attention_head(q, k, v, s, b, topk=C, mode=O.MODE_INFER_HARD)
    causal = np.where(np.tril(np.ones((N, N))) > 0, 0.0, -np.inf)
    ref = _sdpa(q, k, v, causal, 1 / 4.0)
    assert np.allclose(r["O"], ref, atol=1e-12)


def test_train_constant_scores_equals_biased_dense_sdpa():
    # s = const gives log g_m = -log C_i for every historical block: dense causal
    # attention with a -log C_i bias on keys before the current block.
    N, b, d = 50, 8, 16
    q, k, v, _ = _rand_head(N, d, 4)
    s = np.full((N, N), 0.7)
    r = O.sas_attention_head(q, k, v, s, b, topk=64, mode=O.MODE_TRAIN_SOFT)
    mask = np.full((N, N), -np.inf)
    for i in range(N):
        c = i // b
        if c > 0:
            mask[i, :c * b] = -math.log(c)
        mask[i, c * b:i + 1] = 0.0
    ref = _sdpa(q, k, v, mask, 1 / 4.0)
    assert np.allclose(r["O"], ref, atol=1e-12)
    lse_ref = scipy.special.logsumexp(q @ k.T / 4.0 + mask, axis=1)
    assert np.allclose(r["LSE"], lse_ref, atol=1e-12)


def test_k0_equals_block_local_causal_sdpa():
    N, b, d = 45, 8, 16
    q, k, v, rng = _rand_head(N, d, 5)
    s = rng.standard_normal((N, N))
    r = O.sas_attention_head(q, k, v, s, b, topk=0, mode=O.MODE_TRAIN_SOFT)
    blk = np.arange(N) // b
    ok = (blk[:, None] == blk[None, :]) & (np.arange(N)[None, :] <= np.arange(N)[:, None])
    ref = _sdpa(q, k, v, np.where(ok, 0.0, -np.inf), 1 / 4.0)
    assert np.allclose(r["O"], ref, atol=1e-12)
    assert np.all(r["sel_idx"].shape == (N, 0))


@pytest.mark.parametrize("mode", [O.MODE_TRAIN_SOFT, O.MODE_INFER_HARD])
@pytest.mark.parametrize("N,b,K,ties", [(70, 8, 3, False), (64, 16, 2, True), (19, 4, 1, True), (9, 8, 2, False)])
def test_streaming_rows_equal_materialised_matrix(mode, N, b, K, ties):
    q, k, v, rng = _rand_head(N, 8, 6 + N)
    s = rng.integers(0, 3, (N, N)).astype(float) if ties else rng.standard_normal((N, N))
    r = O.sas_attention_head(q, k, v, s, b, K, mode)
    m = O.sas_attention_materialized(q, k, v, s, b, K, mode)
    assert np.allclose(r["O"], m["O"], atol=1e-12)
    assert np.allclose(r["LSE"], m["LSE"], atol=1e-12)
    P = m["P"]
    assert np.allclose(P.sum(axis=1), 1.0)                  # rows sum to 1
    assert P.max() <= 1.0 + 1e-15                           # soft weights bounded (Eq. rank_unbounded)
    assert np.all(P[np.triu_indices(N, 1)] == 0)            # causal


def test_attention_shift_invariant_in_scores():
    # Eq. normalized_log_gate: s -> s + c per row leaves gates, selection and output unchanged.
    N, b = 60, 8
    q, k, v, rng = _rand_head(N, 8, 9)
    s = rng.standard_normal((N, N))
    shift = rng.standard_normal((N, 1)) * 10
    r1 = O.sas_attention_head(q, k, v, s, b, 2)
    r2 = O.sas_attention_head(q, k, v, s + shift, b, 2)
    assert np.array_equal(r1["sel_idx"], r2["sel_idx"])
    assert np.allclose(r1["O"], r2["O"], atol=1e-12)


def test_selected_blocks_change_output_only_through_selected_set():
    # A row's output must not depend on keys/values of blocks it did not select.
    N, b = 48, 8
    q, k, v, rng = _rand_head(N, 8, 10)
    s = rng.standard_normal((N, N))
    i = 47
    r = O.sas_attention_head(q, k, v, s, b, 2, rows=[i])
    sel = set(r["sel_idx"][0])
    k2, v2 = k.copy(), v.copy()
    for m in range(i // b):
        if m not in sel:
            k2[m * b:(m + 1) * b] += 5
            v2[m * b:(m + 1) * b] -= 3
    r2 = O.sas_attention_head(q, k2, v2, s, b, 2, rows=[i])
    assert np.allclose(r["O"], r2["O"], atol=1e-14)


# ---------------------------------------------------------------------- a6

def test_gelu_matches_torch_exact_gelu():
    x = np.linspace(-8, 8, 2001)
    ref = F.gelu(torch.from_numpy(x), approximate="none").numpy()
    assert np.allclose(O.gelu(x), ref, atol=1e-15)
    assert O.gelu(np.array([0.0]))[0] == 0.0
    assert math.isclose(O.gelu(np.array([30.0]))[0], 30.0)


def test_gelu_mlp_matches_torch_linear_pipeline():
    X, W1, W2, b1, b2 = synth.mlp(33, 24, 40, seed=3, std=0.2, bias=True)
    Y = O.gelu_mlp(f64(X), f64(W1), f64(W2), f64(b1), f64(b2))
    h = F.linear(X.double(), W1.double(), b1.double())
    g = F.gelu(h, approximate="none").float().to(torch.bfloat16).double()
    ref = F.linear(g, W2.double(), b2.double()).numpy()
    # the two routes may round a hidden value to different bf16 neighbours
    # (torch rounds via float32): allow a couple of such flips, no more
    assert np.abs(Y - ref).max() < 2e-3
    rows = [0, 5, 32]
    assert np.allclose(O.gelu_mlp(f64(X), f64(W1), f64(W2), f64(b1), f64(b2), rows=rows), Y[rows])


def test_flops_accounting_row():
    # row 130 with b = 64: C_i = 2, current block holds 3 keys (128..130)
    assert O.attention_flops_row(130, 64, 32, 128, 128) == 4 * 128 * (3 + 64 * 2) + 2 * 128 * 2
    assert O.attention_flops_row(64 * 40, 64, 32, 128, 0) == 4 * 128 * (1 + 64 * 32)


# ------------------------------------------------- ablation gate forms (Sec. 4.2)

def test_sigmoid_and_logit_log_gates_closed_forms():
    s = np.array([0.0, 40.0, -40.0, math.log(3.0)])
    lg = O.log_gates(s, O.GATE_SIGMOID)
    assert lg[0] == pytest.approx(math.log(0.5), abs=1e-15)            # sigmoid(0) = 1/2
    assert lg[1] == pytest.approx(0.0, abs=1e-15)                      # sigmoid(s) -> 1
    assert lg[2] == pytest.approx(-40.0, abs=1e-15)                    # log sigmoid(s) ~ s for s << 0
    assert lg[3] == pytest.approx(math.log(0.75), abs=1e-15)           # sigmoid(log 3) = 3/4
    assert np.array_equal(O.log_gates(s, O.GATE_LOGIT), s)             # logit injection: log g = s
    # sigmoid gates are independent: one block's gate ignores the others
    assert O.log_gates(np.array([0.0, 5.0]), O.GATE_SIGMOID)[0] == O.log_gates(np.array([0.0, -5.0]), O.GATE_SIGMOID)[0]


def _one_row_case():
    # Query i = 64 (current block 1, one historical block 0, C_i = 1): all keys
    # zero, so every logit is 0; block 0's 64 values are 1, the query's own
    # value is 0.  With gate g on block 0:
    #   inner: weights g (x64) and 1 -> O = 64 g / (64 g + 1)
    #   outer: probabilities 1/65 each, block 0 rows scaled by g -> O = 64 g / 65
    N, d = 65, 1
    Q = np.ones((N, d))
    K = np.zeros((N, d))
    V = np.zeros((N, d))
    V[:64] = 1.0
    return Q, K, V


@pytest.mark.parametrize("act,s0,g", [(O.GATE_SOFTMAX, 1.7, 1.0), (O.GATE_SIGMOID, 0.0, 0.5),
                                      (O.GATE_SIGMOID, math.log(3.0), 0.75), (O.GATE_LOGIT, math.log(0.25), 0.25)])
def test_inner_and_outer_gate_positions_worked_example(act, s0, g):
    Q, K, V = _one_row_case()
    s = np.full((65, 2), s0)
    inner = O.sas_attention_head(Q, K, V, s, 64, 1, O.MODE_TRAIN_SOFT, rows=[64], act=act, pos=O.GATE_INNER)
    outer = O.sas_attention_head(Q, K, V, s, 64, 1, O.MODE_TRAIN_SOFT, rows=[64], act=act, pos=O.GATE_OUTER)
    assert inner["O"][0, 0] == pytest.approx(64 * g / (64 * g + 1), rel=1e-12)
    assert outer["O"][0, 0] == pytest.approx(64 * g / 65, rel=1e-12)
    assert inner["sel_logg"][0, 0] == pytest.approx(math.log(g), abs=1e-12)
    # inner LSE is over the gated logits, outer LSE over the plain ones (all 0 here)
    assert inner["LSE"][0] == pytest.approx(math.log(64 * g + 1), rel=1e-12)
    assert outer["LSE"][0] == pytest.approx(math.log(65.0), rel=1e-12)
    # the hard (inference) forward ignores the gate in both positions
    hard = O.sas_attention_head(Q, K, V, s, 64, 1, O.MODE_INFER_HARD, rows=[64], act=act, pos=O.GATE_OUTER)
    assert hard["O"][0, 0] == pytest.approx(64 / 65, rel=1e-12)


def test_outer_position_is_affine_in_a_common_gate():
    # With every historical gate equal to g (logit gates, constant scores s =
    # log g, K >= C), the outer output is O_cur + g * O_hist: linear in g, so
    # O(2g) - O(g) = O(g) - O(0) (a gate inside the softmax would not be).
    rng = np.random.default_rng(7)
    N, d = 200, 4
    Q, K, V = (O.round_to_bf16(rng.standard_normal((N, d))) for _ in range(3))
    rows = [70, 150, 199]
    def out(g):
        s = np.full((N, 4), math.log(g)) if g > 0 else np.full((N, 4), -1e300)
        return O.sas_attention_head(Q, K, V, s, 64, 4, rows=rows, act=O.GATE_LOGIT, pos=O.GATE_OUTER)["O"]
    o0, o1, o2 = out(0.0), out(0.8), out(1.6)
    assert np.allclose(o2 - o1, o1 - o0, atol=1e-12)
    inner1 = O.sas_attention_head(Q, K, V, np.full((N, 4), math.log(0.8)), 64, 4, rows=rows,
                                  act=O.GATE_LOGIT, pos=O.GATE_INNER)["O"]
    assert not np.allclose(inner1, o1, atol=1e-3)


def test_ablation_forms_match_materialized_matrix():
    rng = np.random.default_rng(8)
    N, d = 300, 8
    Q, K, V = (O.round_to_bf16(rng.standard_normal((N, d))) for _ in range(3))
    s = rng.standard_normal((N, 5))
    for act in (O.GATE_SOFTMAX, O.GATE_SIGMOID, O.GATE_LOGIT):
        for pos in (O.GATE_INNER, O.GATE_OUTER):
            row = O.sas_attention_head(Q, K, V, s, 64, 2, act=act, pos=pos)
            mat = O.sas_attention_materialized(Q, K, V, s, 64, 2, act=act, pos=pos)
            assert np.allclose(row["O"], mat["O"], atol=1e-12)
            assert np.allclose(row["LSE"], mat["LSE"], atol=1e-12)


# ---------------------------------------------- training scopes (Sec. 4.2, Table 1)

@pytest.mark.parametrize("N,b", [(200, 16), (130, 64)])
def test_full_scope_equals_keep_all_sparse_and_materialised(N, b):
    # Full scope is the sparse oracle with every historical block kept (K >= C_i)
    # and the brute-force matrix with K = C: three separate code paths.
    rng = np.random.default_rng(7)
    d = 16
    Q, K, V = (O.round_to_bf16(rng.standard_normal((N, d))) for _ in range(3))
    s = rng.standard_normal((N, -(-N // b)))
    full = O.sas_attention_full_scope(Q, K, V, s, b)
    C = -(-N // b)
    keep_all = O.sas_attention_head(Q, K, V, s, b, C)
    mat = O.sas_attention_materialized(Q, K, V, s, b, C)
    assert np.allclose(full["O"], keep_all["O"], atol=1e-12)
    assert np.allclose(full["LSE"], keep_all["LSE"], atol=1e-12)
    assert np.allclose(full["O"], mat["O"], atol=1e-12)


def test_full_scope_constant_scores_is_biased_dense_sdpa():
    # constant scores: log g = -log C_i on every historical key, 0 on the causal
    # current block -> torch SDPA with that additive mask
    N, b, d = 192, 32, 16
    rng = np.random.default_rng(8)
    Q, K, V = (O.round_to_bf16(rng.standard_normal((N, d))) for _ in range(3))
    s = np.full((N, N // b), 0.7)
    full = O.sas_attention_full_scope(Q, K, V, s, b)
    mask = np.full((N, N), -np.inf)
    for i in range(N):
        c = i // b
        if c:
            mask[i, :c * b] = -math.log(c)
        mask[i, c * b:i + 1] = 0.0
    ref = F.scaled_dot_product_attention(torch.tensor(Q)[None], torch.tensor(K)[None], torch.tensor(V)[None],
                                         attn_mask=torch.tensor(mask)[None])[0].numpy()
    assert np.allclose(full["O"], ref, atol=1e-10)


def test_noisy_scores_zero_noise_and_shift():
    # full* with zero noise is the sparse form; a constant noise only shifts s,
    # which changes neither the kept set nor log g (Eq. normalized_log_gate)
    rng = np.random.default_rng(9)
    N, b, d, K = 150, 16, 8, 3
    Q, Kk, V = (O.round_to_bf16(rng.standard_normal((N, d))) for _ in range(3))
    s = rng.standard_normal((N, -(-N // b))).astype(np.float32).astype(np.float64)
    base = O.sas_attention_head(Q, Kk, V, s, b, K)
    zero = O.sas_attention_head(Q, Kk, V, O.noisy_scores(s, np.zeros_like(s)), b, K)
    assert np.array_equal(base["sel_idx"], zero["sel_idx"]) and np.allclose(base["O"], zero["O"], atol=0)
    shifted = O.sas_attention_head(Q, Kk, V, O.noisy_scores(s, np.full_like(s, 0.25)), b, K)
    assert np.array_equal(base["sel_idx"], shifted["sel_idx"])
    assert np.allclose(base["O"], shifted["O"], atol=1e-6)


def test_noisy_scores_flip_the_selection():
    # hand example, K = 1: s = (1.0, 1.5) keeps block 1; noise (+1, 0) makes
    # s~ = (2.0, 1.5), which keeps block 0 with log g = 2 - log(e^2 + e^1.5)
    s = np.array([[1.0, 1.5]])
    sn = O.noisy_scores(s, np.array([[1.0, 0.0]]))
    assert O.topk_blocks(s[0], 1).tolist() == [1] and O.topk_blocks(sn[0], 1).tolist() == [0]
    lg = O.log_gates(sn[0])
    assert abs(lg[0] - (2.0 - math.log(math.exp(2.0) + math.exp(1.5)))) < 1e-12
