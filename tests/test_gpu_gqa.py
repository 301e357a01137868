"""GPU parity of the GQA forward (group-shared selection: the G query heads of
a KV group share one score table, one Top-K and one set of tile unions;
Sec. 5.3, Sec. 5 inference implementation) against the fp64 oracle, and
bit-identity with the MHA path run on per-head repeated K, V and scores."""
import numpy as np
import pytest
import torch

from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu

TRAIN, INFER = sas.SAS_MODE_TRAIN_SOFT, sas.SAS_MODE_INFER_HARD


def _inputs(B, Hq, Hkv, N, d, seed, regime="R1"):
    Q = synth.qkv(B, Hq, N, d, seed=seed)[0]
    _, K, V = synth.qkv(B, Hkv, N, d, seed=seed + 100)
    S = synth.scores(B, Hkv, N, -(-N // 64), seed=seed, regime=regime)
    return Q, K, V, S


def _run(B, Hq, Hkv, N, d, topk, mode, Q, K, V, S):
    layer = sas.SasLayer(B, Hq, N, d, topk, mode=mode, Hkv=Hkv)
    dev = torch.device("cuda:0")
    O, LSE, si, sl = layer.attention(*(t.to(dev).contiguous() for t in (Q, K, V)), scores=S.to(dev).contiguous())
    T = -(-N // 128)
    unions = np.array(sas.sas_get_tile_union_counts(layer.h, B * Hkv * T)).reshape(B, Hkv, T)
    status = sas.sas_get_device_status(layer.h)
    layer.close()
    return {"O": O.cpu(), "LSE": LSE.cpu(), "sel_idx": si.cpu(), "sel_logg": sl.cpu(), "unions": unions,
            "status": status}


@pytest.mark.parametrize("B,Hq,Hkv,N,d,topk,mode", [
    (1, 8, 2, 700, 128, 4, TRAIN),     # G = 4, ragged tail, several tiles
    (2, 6, 3, 389, 128, 2, INFER),     # G = 2, inference form
    (1, 4, 1, 517, 64, 3, TRAIN),      # MQA (one KV head), d = 64
])
def test_gqa_matches_oracle(B, Hq, Hkv, N, d, topk, mode):
    Q, K, V, S = _inputs(B, Hq, Hkv, N, d, seed=Hq + N)
    g = _run(B, Hq, Hkv, N, d, topk, mode, Q, K, V, S)
    assert g["status"] == 0
    ref = OR.sas_attention_gqa(P.f64(Q), P.f64(K), P.f64(V), 64, topk, P.f64(S), mode=mode)
    G = Hq // Hkv
    for bi in range(B):
        for hi in range(Hq):
            r = ref[(bi, hi)]
            gk = hi // G
            if hi % G == 0:   # the group's kept lists, once per group
                gi = g["sel_idx"][bi, gk].numpy()[:, :topk]
                P.check_selection_rows(gi, P.f64(S[bi, gk]), np.arange(N), topk)
                lg = g["sel_logg"][bi, gk].numpy()[:, :topk]
                assert np.abs(lg - r["sel_logg"]).max(initial=0) <= P.LOGG_MAX_ABS
                assert np.array_equal(g["unions"][bi, gk], P.oracle_union_counts(gi, N, topk))
            P.compare_o(P.f64(g["O"][bi, hi]), r["O"], f"O[{bi},{hi}]")
            assert np.abs(g["LSE"][bi, hi].numpy() - r["LSE"]).max() <= P.LSE_MAX_ABS


def test_gqa_is_bit_identical_to_mha_on_repeated_inputs():
    B, Hq, Hkv, N, d, topk = 2, 8, 2, 1100, 128, 5
    G = Hq // Hkv
    Q, K, V, S = _inputs(B, Hq, Hkv, N, d, seed=3)
    g = _run(B, Hq, Hkv, N, d, topk, TRAIN, Q, K, V, S)
    rep = lambda t: t.repeat_interleave(G, dim=1)
    m = _run(B, Hq, Hq, N, d, topk, TRAIN, Q, rep(K), rep(V), rep(S))
    assert g["status"] == 0 and m["status"] == 0
    assert torch.equal(g["O"], m["O"])
    assert torch.equal(g["LSE"], m["LSE"])
    assert torch.equal(rep(g["sel_idx"]), m["sel_idx"])
    assert torch.equal(rep(g["sel_logg"]), m["sel_logg"])


def test_qwen3_4b_shaped_prefill_sampled_rows():
    # Hq = 32, Hkv = 8 (G = 4), d = 128, K = 32, 8192 tokens: sampled rows of two heads
    B, Hq, Hkv, N, d, topk = 1, 32, 8, 8192, 128, 32
    Q, K, V, S = _inputs(B, Hq, Hkv, N, d, seed=5)
    g = _run(B, Hq, Hkv, N, d, topk, TRAIN, Q, K, V, S)
    assert g["status"] == 0
    rows = P.sample_rows(N, 128, seed=1)
    heads = [(0, 5), (0, 30)]
    ref = OR.sas_attention_gqa(P.f64(Q), P.f64(K), P.f64(V), 64, topk, P.f64(S), heads=heads, rows=rows)
    for (bi, hi), r in ref.items():
        P.compare_o(P.f64(g["O"][bi, hi])[rows], r["O"], f"O[{bi},{hi}]")
        assert np.abs(g["LSE"][bi, hi].numpy()[rows] - r["LSE"]).max() <= P.LSE_MAX_ABS
        gi = g["sel_idx"][bi, hi // 4].numpy()[rows][:, :topk]
        P.check_selection_rows(gi, P.f64(S[bi, hi // 4])[rows], rows, topk)


@pytest.mark.parametrize("G,Hkv,N,topk", [
    (2, 2, 700, 4),     # 64 tokens of 2 heads per tile
    (8, 1, 517, 3),     # 16 tokens of 8 heads
    (16, 1, 389, 2),    # 8 tokens of 16 heads
])
def test_head_packed_tiles_match_oracle(G, Hkv, N, topk):
    # tiles of 128 / G tokens x the G heads of a KV group (one kept list per token):
    # every row against the oracle, and the tile count of the work the kernel did
    Hq = G * Hkv
    Q, K, V, S = _inputs(1, Hq, Hkv, N, 128, seed=G + N)
    layer = sas.SasLayer(1, Hq, N, 128, topk, Hkv=Hkv)
    dev = torch.device("cuda:0")
    O, LSE, si, sl = layer.attention(*(t.to(dev).contiguous() for t in (Q, K, V)), scores=S.to(dev).contiguous())
    tiles, blocks = sas.sas_get_attention_work(layer.h)
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    R = 128 // G
    assert tiles == Hkv * -(-N // R)
    assert blocks >= tiles   # every tile visits at least its diagonal block
    ref = OR.sas_attention_gqa(P.f64(Q), P.f64(K), P.f64(V), 64, topk, P.f64(S))
    for hi in range(Hq):
        r = ref[(0, hi)]
        P.compare_o(P.f64(O[0, hi].cpu()), r["O"], f"O[0,{hi}]")
        assert np.abs(LSE[0, hi].cpu().numpy() - r["LSE"]).max() <= P.LSE_MAX_ABS


@pytest.mark.parametrize("B,Hq,Hkv,N,d,d_sel,topk", [
    (1, 8, 2, 1000, 128, 128, 4),     # G = 4
    (2, 4, 2, 700, 64, 64, 3),        # G = 2, d = 64
])
def test_gqa_learned_selector_exact_inputs(B, Hq, Hkv, N, d, d_sel, topk):
    # integer Q, K and {-1, 0, 1} projections: every selector sum is exact in fp32,
    # so the group gate query's kept sets must equal the oracle's on every row
    G = Hq // Hkv
    Q = synth.integer_selector_inputs(B, Hq, N, d, d_sel, seed=Hq)[0]
    _, K, V, _, _ = synth.integer_selector_inputs(B, Hkv, N, d, d_sel, seed=Hq + 1)
    Wq, Wk = synth.decode_selector_weights(Hkv, G, d, d_sel, seed=Hq, exact=True)
    dev = torch.device("cuda:0")
    layer = sas.SasLayer(B, Hq, N, d, topk, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d_sel, Hkv=Hkv)
    O, LSE, si, sl = layer.attention(*(t.to(dev).contiguous() for t in (Q, K, V)), Wq=Wq.to(dev), Wk=Wk.to(dev))
    T = -(-N // 128)
    unions = np.array(sas.sas_get_tile_union_counts(layer.h, B * Hkv * T)).reshape(B, Hkv, T)
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    ref = OR.sas_attention_gqa(P.f64(Q), P.f64(K), P.f64(V), 64, topk, Wq=P.f64(Wq), Wk=P.f64(Wk))
    for bi in range(B):
        for g in range(Hkv):
            s = OR.selector_scores_group(P.f64(Q[bi, g * G:(g + 1) * G]), P.f64(K[bi, g]), P.f64(Wq[g]),
                                         P.f64(Wk[g]), 64)
            gi = si[bi, g].cpu().numpy()[:, :topk]
            P.check_selection_rows(gi, s, np.arange(N), topk)
            assert np.array_equal(unions[bi, g], P.oracle_union_counts(gi, N, topk))
            lg = sl[bi, g].cpu().numpy()[:, :topk]
            assert np.abs(lg - ref[(bi, g * G)]["sel_logg"]).max(initial=0) <= P.LOGG_MAX_ABS
        for hi in range(Hq):
            r = ref[(bi, hi)]
            P.compare_o(P.f64(O[bi, hi].cpu()), r["O"], f"O[{bi},{hi}]")
            assert np.abs(LSE[bi, hi].cpu().numpy() - r["LSE"]).max() <= P.LSE_MAX_ABS
