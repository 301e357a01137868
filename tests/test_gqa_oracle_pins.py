"""Pins of the GQA oracle (group-shared selection, Sec. 5.3 / Sec. 5 inference
implementation): G = 1 is the MHA oracle, a GQA layer equals the MHA oracle
on K, V and scores repeated per query head, every head of a group keeps the
same blocks, and one group's heads agree with the brute-force materialised
attention of that group.  CPU only."""
import numpy as np
import pytest

from oracle import sas_oracle as O


def _inputs(B, Hq, Hkv, N, d, seed):
    rng = np.random.default_rng(seed)
    C = -(-N // 8)
    Q = rng.standard_normal((B, Hq, N, d))
    K = rng.standard_normal((B, Hkv, N, d))
    V = rng.standard_normal((B, Hkv, N, d))
    s = rng.standard_normal((B, Hkv, N, C))
    return Q, K, V, s


def test_single_head_groups_are_the_mha_oracle():
    Q, K, V, s = _inputs(2, 3, 3, 37, 5, 0)
    a = O.sas_attention_gqa(Q, K, V, 8, 2, s)
    m = O.sas_attention(Q, K, V, 8, 2, scores=s)
    for key in m:
        for f in ("O", "LSE", "sel_idx", "sel_logg"):
            assert np.array_equal(a[key][f], m[key][f])


@pytest.mark.parametrize("G,mode", [(2, O.MODE_TRAIN_SOFT), (4, O.MODE_INFER_HARD), (3, O.MODE_TRAIN_SOFT)])
def test_gqa_equals_mha_on_repeated_kv_and_scores(G, mode):
    B, Hkv, N, d = 2, 2, 45, 4
    Q, K, V, s = _inputs(B, G * Hkv, Hkv, N, d, G)
    a = O.sas_attention_gqa(Q, K, V, 8, 2, s, mode=mode)
    rep = lambda x: np.repeat(x, G, axis=1)     # query head h reads group h // G
    m = O.sas_attention(Q, rep(K), rep(V), 8, 2, mode=mode, scores=rep(s))
    for key in m:
        for f in ("O", "LSE", "sel_idx", "sel_logg"):
            assert np.array_equal(a[key][f], m[key][f]), (key, f)


def test_heads_of_a_group_keep_the_same_blocks_and_others_may_differ():
    G, Hkv, N = 4, 2, 64
    Q, K, V, s = _inputs(1, G * Hkv, Hkv, N, 3, 7)
    a = O.sas_attention_gqa(Q, K, V, 8, 2, s)
    for g in range(Hkv):
        ref = a[(0, g * G)]["sel_idx"]
        for h in range(g * G + 1, (g + 1) * G):
            assert np.array_equal(a[(0, h)]["sel_idx"], ref)
            assert np.array_equal(a[(0, h)]["sel_logg"], a[(0, g * G)]["sel_logg"])
    # the two groups' scores differ, so (with these seeds) their kept sets do
    assert not np.array_equal(a[(0, 0)]["sel_idx"], a[(0, G)]["sel_idx"])


def test_group_heads_match_the_materialised_attention_of_the_group():
    G, Hkv, N, d = 2, 2, 33, 4
    Q, K, V, s = _inputs(1, G * Hkv, Hkv, N, d, 11)
    a = O.sas_attention_gqa(Q, K, V, 8, 3, s)
    for h in range(G * Hkv):
        g = h // G
        ref = O.sas_attention_materialized(Q[0, h], K[0, g], V[0, g], s[0, g], 8, 3)
        assert np.allclose(a[(0, h)]["O"], ref["O"], atol=1e-12)
        assert np.allclose(a[(0, h)]["LSE"], ref["LSE"], atol=1e-12)


def test_query_heads_must_fill_whole_groups():
    Q, K, V, s = _inputs(1, 3, 2, 16, 2, 1)
    with pytest.raises(ValueError):
        O.sas_attention_gqa(Q, K, V, 8, 1, s)


def test_group_gate_query_reduces_to_the_head_selector():
    # G = 1: the group gate query is the per-head selector
    rng = np.random.default_rng(3)
    N, d, ds = 70, 6, 4
    Q, K = rng.standard_normal((1, N, d)), rng.standard_normal((N, d))
    Wq, Wk = rng.standard_normal((ds, d)), rng.standard_normal((ds, d))
    assert np.array_equal(O.selector_scores_group(Q, K, Wq, Wk, 8), O.selector_scores(Q[0], K, Wq, Wk, 8))
    # G = 3 with weight only on head 1's slice: head 1's per-head selector, exactly
    Qg = rng.standard_normal((3, N, d))
    Wg = np.zeros((ds, 3 * d))
    Wg[:, d:2 * d] = Wq
    assert np.array_equal(O.selector_scores_group(Qg, K, Wg, Wk, 8), O.selector_scores(Qg[1], K, Wq, Wk, 8))


def test_group_gate_query_with_equal_slices_is_the_sum_of_the_heads():
    # Wq_g = [W W] makes q~ = bf16(W (q_0 + q_1)): the selector of the summed queries
    rng = np.random.default_rng(4)
    N, d, ds = 64, 4, 4
    Qg, K = rng.standard_normal((2, N, d)), rng.standard_normal((N, d))
    W, Wk = rng.standard_normal((ds, d)), rng.standard_normal((ds, d))
    a = O.selector_scores_group(Qg, K, np.concatenate([W, W], axis=1), Wk, 8)
    b = O.selector_scores(Qg[0] + Qg[1], K, W, Wk, 8)
    assert np.allclose(a, b, rtol=0, atol=1e-12)


def test_learned_gqa_uses_one_table_per_group():
    rng = np.random.default_rng(5)
    B, Hkv, G, N, d, ds = 1, 2, 2, 48, 4, 4
    Q = rng.standard_normal((B, Hkv * G, N, d))
    K, V = rng.standard_normal((B, Hkv, N, d)), rng.standard_normal((B, Hkv, N, d))
    Wq, Wk = rng.standard_normal((Hkv, ds, G * d)), rng.standard_normal((Hkv, ds, d))
    a = O.sas_attention_gqa(Q, K, V, 8, 2, Wq=Wq, Wk=Wk)
    for g in range(Hkv):
        s = O.selector_scores_group(Q[0, g * G:(g + 1) * G], K[0, g], Wq[g], Wk[g], 8)
        ref = O.sas_attention_gqa(Q, K, V, 8, 2, scores=np.broadcast_to(s, (B, Hkv) + s.shape).copy())
        for h in range(g * G, (g + 1) * G):
            assert np.array_equal(a[(0, h)]["O"], ref[(0, h)]["O"])
            assert np.array_equal(a[(0, h)]["sel_idx"], ref[(0, h)]["sel_idx"])


def test_group_gate_query_agrees_with_the_decode_oracle():
    # the decode step (its own oracle module) reads the group gate query the same
    # way: its scores for the newest token are the last prefill row's
    from oracle import decode_oracle as D
    rng = np.random.default_rng(6)
    G, n, d, ds, b = 4, 200, 8, 4, 16
    Qg, K, V = rng.standard_normal((G, n, d)), rng.standard_normal((n, d)), rng.standard_normal((n, d))
    Wq, Wk = rng.standard_normal((ds, G * d)), rng.standard_normal((ds, d))
    pre = O.selector_scores_group(Qg, K, Wq, Wk, b)
    dec = D.decode_group(Qg[:, n - 1, :], K, V, Wq, Wk, b, 3)
    C = (n - 1) // b
    assert np.allclose(pre[n - 1, :C], dec["scores"], rtol=0, atol=1e-12)
