"""Pins of the packed variable-length oracle (cu_seqlens offsets; the authors'
kernel packs sequences, which the pseudocode omits): equal-length packing
equals the batched oracle, a sequence's first n tokens give the same outputs
as the sequence cut to n tokens (causality), a sequence does not see its
neighbours, and its block partition starts at its own first token whatever
its offset in the pack.  CPU only."""
import numpy as np
import pytest

from oracle import sas_oracle as O


def _packed(lens, Hq, Hkv, d, seed, C=None):
    rng = np.random.default_rng(seed)
    total = int(sum(lens))
    C = C or -(-max(lens) // 8)
    Q = rng.standard_normal((Hq, total, d))
    K = rng.standard_normal((Hkv, total, d))
    V = rng.standard_normal((Hkv, total, d))
    s = rng.standard_normal((Hkv, total, C))
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    return Q, K, V, s, cu


@pytest.mark.parametrize("mode", [O.MODE_TRAIN_SOFT, O.MODE_INFER_HARD])
def test_equal_lengths_pack_equals_the_batched_oracle(mode):
    S, H, n, d = 3, 2, 29, 4
    Q, K, V, s, cu = _packed([n] * S, H, H, d, 0)
    v = O.sas_attention_varlen(Q, K, V, cu, 8, 2, s, mode=mode)
    # the same data laid out as a [B = S, H, n, d] batch
    bat = lambda x: x.reshape(x.shape[0], S, n, -1).transpose(1, 0, 2, 3)
    m = O.sas_attention(bat(Q), bat(K), bat(V), 8, 2, mode=mode, scores=bat(s))
    for bi in range(S):
        for hi in range(H):
            rows = slice(cu[bi], cu[bi + 1])
            assert np.array_equal(v["O"][hi, rows], m[(bi, hi)]["O"])
            assert np.array_equal(v["LSE"][hi, rows], m[(bi, hi)]["LSE"])
            assert np.array_equal(v["sel_idx"][hi, rows], m[(bi, hi)]["sel_idx"])


def test_prefix_of_a_sequence_equals_the_shorter_sequence():
    Q, K, V, s, cu = _packed([41, 70], 2, 1, 3, 1)
    full = O.sas_attention_varlen(Q, K, V, cu, 8, 2, s)
    # cut the second sequence to its first 50 tokens
    keep = np.r_[0:41, 41:91]
    cut = O.sas_attention_varlen(Q[:, keep], K[:, keep], V[:, keep], [0, 41, 91], 8, 2, s[:, keep])
    assert np.array_equal(cut["O"], full["O"][:, keep])
    assert np.array_equal(cut["sel_idx"], full["sel_idx"][:, keep])


def test_sequences_do_not_see_each_other():
    Q, K, V, s, cu = _packed([37, 53, 20], 2, 2, 3, 2)
    a = O.sas_attention_varlen(Q, K, V, cu, 8, 3, s)
    K2, V2, s2 = K.copy(), V.copy(), s.copy()
    K2[:, 37:90] += 5.0      # change the middle sequence only
    V2[:, 37:90] -= 3.0
    s2[:, 37:90] *= -1.0
    b = O.sas_attention_varlen(Q, K2, V2, cu, 8, 3, s2)
    for rows in (slice(0, 37), slice(90, 110)):
        assert np.array_equal(a["O"][:, rows], b["O"][:, rows])
        assert np.array_equal(a["sel_idx"][:, rows], b["sel_idx"][:, rows])
    assert not np.allclose(a["O"][:, 37:90], b["O"][:, 37:90])


def test_block_partition_starts_at_each_sequence_start():
    # the same 45-token sequence after a 13-token one and alone: identical
    # outputs, although 13 is not a multiple of the block size
    Q, K, V, s, cu = _packed([13, 45], 2, 2, 3, 3)
    pack = O.sas_attention_varlen(Q, K, V, cu, 8, 2, s)
    alone = O.sas_attention_varlen(Q[:, 13:], K[:, 13:], V[:, 13:], [0, 45], 8, 2, s[:, 13:])
    assert np.array_equal(pack["O"][:, 13:], alone["O"])
    assert np.array_equal(pack["sel_idx"][:, 13:], alone["sel_idx"])
    # and a token's blocks are counted from its own sequence: token 8 of the
    # second sequence has exactly one historical block (block 0 of that sequence)
    assert (pack["sel_idx"][:, 13 + 8] >= 0).sum(axis=1).tolist() == [1, 1]


def test_gqa_packing_and_empty_sequences_and_bad_offsets():
    Q, K, V, s, cu = _packed([30, 0, 21], 4, 2, 3, 4)
    v = O.sas_attention_varlen(Q, K, V, cu, 8, 2, s)
    g = O.sas_attention_gqa(Q[None, :, :30], K[None, :, :30], V[None, :, :30], 8, 2, s[None, :, :30])
    for h in range(4):
        assert np.array_equal(v["O"][h, :30], g[(0, h)]["O"])
    with pytest.raises(ValueError):
        O.sas_attention_varlen(Q, K, V, [0, 40, 30, 51], 8, 2, s)
    with pytest.raises(ValueError):
        O.sas_attention_varlen(Q, K, V, [1, 30, 51], 8, 2, s)


def test_learned_selector_pack_equals_the_batched_learned_oracle():
    # equal lengths, the learned selector (group gate query, G = 2): the pack equals
    # the batched GQA oracle, whose block summaries are per batch element
    S, Hkv, G, n, d, ds = 2, 1, 2, 70, 4, 4
    rng = np.random.default_rng(31)
    Q = rng.standard_normal((Hkv * G, S * n, d))
    K, V = rng.standard_normal((Hkv, S * n, d)), rng.standard_normal((Hkv, S * n, d))
    Wq, Wk = rng.standard_normal((Hkv, ds, G * d)), rng.standard_normal((Hkv, ds, d))
    cu = np.array([0, n, 2 * n])
    v = O.sas_attention_varlen(Q, K, V, cu, 8, 2, Wq=Wq, Wk=Wk)
    bat = lambda x: x.reshape(x.shape[0], S, n, -1).transpose(1, 0, 2, 3)
    m = O.sas_attention_gqa(bat(Q), bat(K), bat(V), 8, 2, Wq=Wq, Wk=Wk)
    for bi in range(S):
        for h in range(Hkv * G):
            assert np.array_equal(v["O"][h, bi * n:(bi + 1) * n], m[(bi, h)]["O"])
            assert np.array_equal(v["sel_idx"][h // G, bi * n:(bi + 1) * n], m[(bi, h)]["sel_idx"])


def test_learned_selector_summaries_stay_within_the_sequence():
    # changing the keys of the first sequence leaves the second one's selection alone
    rng = np.random.default_rng(32)
    Q = rng.standard_normal((1, 150, 4))
    K, V = rng.standard_normal((1, 150, 4)), rng.standard_normal((1, 150, 4))
    Wq, Wk = rng.standard_normal((1, 4, 4)), rng.standard_normal((1, 4, 4))
    cu = [0, 61, 150]
    a = O.sas_attention_varlen(Q, K, V, cu, 8, 2, Wq=Wq, Wk=Wk)
    K2 = K.copy()
    K2[:, :61] *= -2.0
    b = O.sas_attention_varlen(Q, K2, V, cu, 8, 2, Wq=Wq, Wk=Wk)
    assert np.array_equal(a["sel_idx"][:, 61:], b["sel_idx"][:, 61:])
    assert np.array_equal(a["O"][:, 61:], b["O"][:, 61:])
    assert not np.array_equal(a["O"][:, :61], b["O"][:, :61])
