"""Pins of the decode-step oracle (Alg. 2 with per-group selection) against
what the paper and the mathematics fix: a hand-derived worked example, the
reduction to the prefill oracle's last row, dense attention from torch, the
keep-all special case, the head order of the group gate query, and the paging
indirection.  CPU only."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import decode_oracle as D
from oracle import sas_oracle as O


def _rand(shape, rng, scale=1.0):
    return O.round_to_bf16(scale * rng.standard_normal(shape))


def test_worked_example_two_heads_one_kept_block():
    # b = 64, d = d_s = 2, G = 2, Wk = I, Wq_g = [I, I] (q~ = q_0 + q_1), K = 1.
    # Blocks 0, 1, 2 hold keys (1,0), (0,1), (-1,0) and values (1,0), (0,0),
    # (0,0); the new token (position 192, block 3) has key (0,0), value (0,1).
    # q_0 = (2,0), q_1 = (0,0): q~ = (2,0), s = (2, 0, -2)/sqrt(2), I = {0}.
    # Head 0 sees 64 keys with logit 2/sqrt(2) = sqrt(2) and one with 0;
    # head 1 sees 65 zero logits.
    b, n = 64, 193
    K = np.zeros((n, 2))
    V = np.zeros((n, 2))
    K[0:64] = (1, 0)
    K[64:128] = (0, 1)
    K[128:192] = (-1, 0)
    V[0:64] = (1, 0)
    V[192] = (0, 1)
    q = np.array([[2.0, 0.0], [0.0, 0.0]])
    Wq = np.hstack([np.eye(2), np.eye(2)])
    r = D.decode_group(q, K, V, Wq, np.eye(2), b, topk=1)
    assert list(r["sel"]) == [0]
    assert np.allclose(r["scores"], np.array([2.0, 0.0, -2.0]) / math.sqrt(2), atol=0)
    e = math.exp(math.sqrt(2))
    assert np.allclose(r["O"][0], [64 * e / (64 * e + 1), 1 / (64 * e + 1)], atol=1e-15)
    assert np.allclose(r["O"][1], [64 / 65, 1 / 65], atol=1e-15)
    assert np.allclose(r["LSE"], [math.log(64 * e + 1), math.log(65)], atol=1e-14)


def test_first_token_attends_to_itself():
    rng = np.random.default_rng(1)
    K, V = _rand((1, 8), rng), _rand((1, 8), rng)
    q = _rand((3, 8), rng)
    r = D.decode_group(q, K, V, _rand((4, 24), rng), _rand((4, 8), rng), 8, topk=2)
    assert r["sel"].size == 0 and r["scores"].size == 0
    assert np.allclose(r["O"], np.repeat(V, 3, axis=0), atol=0)
    assert np.allclose(r["LSE"], (q @ K[0]) / math.sqrt(8), atol=1e-14)


@pytest.mark.parametrize("n", [1, 8, 9, 16, 17, 43, 64, 70])
@pytest.mark.parametrize("topk", [0, 1, 3])
def test_single_head_group_equals_last_row_of_prefill_oracle(n, topk):
    # G = 1: the decode step of token n-1 is row n-1 of the causal prefill in
    # inference mode (Alg. 2), with the same selector.
    rng = np.random.default_rng(n * 10 + topk)
    b, d, ds = 8, 16, 8
    Q, K, V = _rand((n, d), rng), _rand((n, d), rng), _rand((n, d), rng)
    Wq, Wk = _rand((ds, d), rng, 0.3), _rand((ds, d), rng, 0.3)
    s = O.selector_scores(Q, K, Wq, Wk, b)
    if s.shape[1] < O.num_blocks(n, b):
        s = np.pad(s, ((0, 0), (0, O.num_blocks(n, b) - s.shape[1])))
    ref = O.sas_attention_head(Q, K, V, s, b, topk, O.MODE_INFER_HARD, rows=[n - 1])
    r = D.decode_group(Q[n - 1:n], K, V, Wq, Wk, b, topk)
    assert np.array_equal(r["sel"], ref["sel_idx"][0][ref["sel_idx"][0] >= 0])
    assert np.allclose(r["O"][0], ref["O"][0], atol=1e-13)
    assert np.allclose(r["LSE"][0], ref["LSE"][0], atol=1e-13)


@pytest.mark.parametrize("n", [1, 30, 64, 65])
def test_dense_decode_equals_torch_attention(n):
    rng = np.random.default_rng(n)
    G, d = 4, 16
    q, K, V = _rand((G, d), rng), _rand((n, d), rng), _rand((n, d), rng)
    r = D.decode_group(q, K, V, _rand((8, G * d), rng), _rand((8, d), rng), 8, topk=1, dense=True)
    t = lambda a: torch.from_numpy(a)[None]
    ref = F.scaled_dot_product_attention(t(q), t(K), t(V), scale=1 / 4.0)[0].numpy()
    assert np.allclose(r["O"], ref, atol=1e-13)
    lse = torch.logsumexp(torch.from_numpy(q @ K.T) / 4.0, dim=-1).numpy()
    assert np.allclose(r["LSE"], lse, atol=1e-13)


def test_keep_all_equals_dense():
    rng = np.random.default_rng(7)
    G, d, b, n = 2, 8, 8, 45           # C = 5 historical blocks
    q, K, V = _rand((G, d), rng), _rand((n, d), rng), _rand((n, d), rng)
    Wq, Wk = _rand((4, G * d), rng), _rand((4, d), rng)
    sparse = D.decode_group(q, K, V, Wq, Wk, b, topk=5)
    dense = D.decode_group(q, K, V, Wq, Wk, b, topk=0, dense=True)
    assert list(sparse["sel"]) == [0, 1, 2, 3, 4]
    assert np.allclose(sparse["O"], dense["O"], atol=1e-15)


@pytest.mark.parametrize("j", [0, 1, 2])
def test_group_gate_query_head_order(j):
    # Wq_g nonzero only on head j's slice: the group selects exactly what the
    # single-head selector of head j selects (pins the head-major concatenation).
    rng = np.random.default_rng(20 + j)
    G, d, ds, b, n = 3, 8, 8, 8, 77
    q, K, V = _rand((G, d), rng), _rand((n, d), rng), _rand((n, d), rng)
    W, Wk = _rand((ds, d), rng, 0.5), _rand((ds, d), rng, 0.5)
    Wq = np.zeros((ds, G * d))
    Wq[:, j * d:(j + 1) * d] = W
    r = D.decode_group(q, K, V, Wq, Wk, b, topk=3)
    s_head = O.selector_scores(q[j:j + 1], K, W, Wk, b)[0][:(n - 1) // b]
    assert np.allclose(r["scores"], s_head, atol=1e-15)
    assert np.array_equal(r["sel"], O.topk_blocks(s_head, 3))


def test_selection_ties_go_to_lower_block():
    # all blocks identical -> all scores equal -> the K lowest blocks
    G, d, b, n = 1, 4, 8, 8 * 6 + 3
    K = np.tile(np.array([1.0, 0.5, -1.0, 0.25]), (n, 1))
    V = np.arange(n * d, dtype=np.float64).reshape(n, d) / 100
    q = np.array([[1.0, 1.0, 1.0, 1.0]])
    r = D.decode_group(q, K, V, np.eye(4), np.eye(4), b, topk=2)
    assert list(r["sel"]) == [0, 1]
    assert np.all(r["scores"] == r["scores"][0])


def test_paged_cache_equals_contiguous_context():
    rng = np.random.default_rng(5)
    B, Hkv, G, d, ds, b, topk = 3, 2, 2, 8, 8, 8, 2
    lens = [1, 33, 57]
    max_blocks = 8
    P = B * max_blocks
    perm = rng.permutation(P)
    table = perm.reshape(B, max_blocks)
    Kc, Vc = _rand((P, Hkv, b, d), rng), _rand((P, Hkv, b, d), rng)
    q = _rand((B, Hkv * G, d), rng)
    Wq, Wk = _rand((Hkv, ds, G * d), rng, 0.4), _rand((Hkv, ds, d), rng, 0.4)
    r = D.decode_step(q, Kc, Vc, table, lens, Wq, Wk, b, topk)
    for bi in range(B):
        for g in range(Hkv):
            Kx = np.concatenate([Kc[table[bi, m], g] for m in range(max_blocks)])[:lens[bi]]
            Vx = np.concatenate([Vc[table[bi, m], g] for m in range(max_blocks)])[:lens[bi]]
            ref = D.decode_group(q[bi, g * G:(g + 1) * G], Kx, Vx, Wq[g], Wk[g], b, topk)
            assert np.allclose(r["O"][bi, g * G:(g + 1) * G], ref["O"], atol=0)
            got = r["sel_idx"][bi, g]
            assert np.array_equal(got[got >= 0], ref["sel"])


def test_decode_bytes_accounting():
    # n = 4097: C = 64 historical blocks, current block holds one token
    by = D.decode_bytes_per_group(4097, 64, 32, 128, 128, 4)
    attended = 32 * 64 + 1
    expect = 4 * 2 * 128 + 2 * 4 * 128 + 2 * 128 * 512 + 2 * 64 * 128 + 4 * attended * 128 + 2 * 4 * 128
    assert by == expect
    dense = D.decode_bytes_per_group(4097, 64, 32, 128, 128, 4, dense=True)
    assert dense == 4 * 2 * 128 + 2 * 4 * 128 + 4 * 4097 * 128 + 2 * 4 * 128
