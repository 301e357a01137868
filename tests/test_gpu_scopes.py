"""GPU parity of the training scopes of Sec. 4.2 (Table 1 settings 9-11) against
the fp64 oracle, through the C ABI:
  * full scope (SAS_SCOPE_FULL): every historical block gated, no Top-K --
    checked against oracle.sas_attention_full_scope, including N >= 8192 where
    rows have more than 64 historical blocks;
  * full* (sas_attention_fwd_noisy): noise added to the scores before the
    gate and the Top-K -- zero noise is bit-identical to the sparse path,
    noisy selections match the oracle on the fp32 sum s + eps."""
import numpy as np
import pytest
import torch

from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
TRAIN, INFER = sas.SAS_MODE_TRAIN_SOFT, sas.SAS_MODE_INFER_HARD


def _full_given(B, H, N, d, mode=TRAIN, rows=None, seed=0, Hkv=0):
    Hk = Hkv or H
    Q = synth.qkv(B, H, N, d, seed=seed)[0]
    _, K, V = synth.qkv(B, Hk, N, d, seed=seed + 100)
    S = synth.scores(B, Hk, N, -(-N // 64), seed=seed, regime="R1")
    layer = sas.SasLayer(B, H, N, d, 4, mode=mode, selector=sas.SAS_SEL_SCORES_GIVEN, Hkv=Hkv,
                         scope=sas.SAS_SCOPE_FULL)
    O, LSE, si, sl = layer.attention(Q.to(DEV), K.to(DEV), V.to(DEV), scores=S.to(DEV))
    torch.cuda.synchronize()
    assert si is None and sl is None
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    G = H // Hk
    rr = np.arange(N) if rows is None else rows
    for bi in range(B):
        for hi in range(H):
            g = hi // G
            if mode == TRAIN:
                ref = OR.sas_attention_full_scope(P.f64(Q[bi, hi]), P.f64(K[bi, g]), P.f64(V[bi, g]),
                                                  P.f64(S[bi, g]), 64, rows=rr)
            else:   # no gates: dense causal attention (the keep-all inference form)
                ref = OR.sas_attention_head(P.f64(Q[bi, hi]), P.f64(K[bi, g]), P.f64(V[bi, g]), P.f64(S[bi, g]),
                                            64, N, INFER, rows=rr)
            P.compare_o(P.f64(O[bi, hi].cpu())[rr], ref["O"], f"O[{bi},{hi}]")
            assert np.abs(LSE[bi, hi].cpu().numpy()[rr] - ref["LSE"]).max() <= P.LSE_MAX_ABS


@pytest.mark.parametrize("d", [128, 64])
def test_full_scope_given_scores_ragged(d):
    _full_given(1, 2, 1000, d, seed=d)


def test_full_scope_inference_mode_is_dense_causal():
    _full_given(1, 1, 700, 64, mode=INFER, seed=3)


def test_full_scope_gqa():
    _full_given(1, 4, 900, 128, seed=4, Hkv=2)


def test_full_scope_long_history_sampled():
    # N = 8192 + 40: rows have up to 128 historical blocks, far more than any Top-K
    N = 8192 + 40
    _full_given(1, 2, N, 128, rows=P.sample_rows(N, n_random=128), seed=5)


def test_full_scope_learned_selector_exact_inputs():
    B, H, N, d = 1, 2, 1500, 128
    Q, K, V, Wq, Wk = synth.integer_selector_inputs(B, H, N, d, d, seed=6)
    layer = sas.SasLayer(B, H, N, d, 4, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d, scope=sas.SAS_SCOPE_FULL)
    O, LSE, _, _ = layer.attention(Q.to(DEV), K.to(DEV), V.to(DEV), Wq=Wq.to(DEV), Wk=Wk.to(DEV))
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    for hi in range(H):
        s = P.oracle_scores(Q, K, Wq, Wk, 0, hi)
        ref = OR.sas_attention_full_scope(P.f64(Q[0, hi]), P.f64(K[0, hi]), P.f64(V[0, hi]), s, 64)
        P.compare_o(P.f64(O[0, hi].cpu()), ref["O"], f"O[0,{hi}]")
        assert np.abs(LSE[0, hi].cpu().numpy() - ref["LSE"]).max() <= P.LSE_MAX_ABS


def test_full_scope_learned_selector_long_history_sampled():
    N = 8192 + 512
    Q, K, V = synth.qkv(1, 2, N, 128, seed=7, regime="R2")
    Wq, Wk = synth.selector_weights(2, 128, 128, seed=7)
    layer = sas.SasLayer(1, 2, N, 128, 32, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=128, scope=sas.SAS_SCOPE_FULL)
    O, LSE, _, _ = layer.attention(Q.to(DEV), K.to(DEV), V.to(DEV), Wq=Wq.to(DEV), Wk=Wk.to(DEV))
    torch.cuda.synchronize()
    layer.close()
    rows = P.sample_rows(N, n_random=128)
    for hi in range(2):
        s = P.oracle_scores(Q, K, Wq, Wk, 0, hi)
        ref = OR.sas_attention_full_scope(P.f64(Q[0, hi]), P.f64(K[0, hi]), P.f64(V[0, hi]), s, 64, rows=rows)
        P.compare_o(P.f64(O[0, hi].cpu())[rows], ref["O"], f"O[0,{hi}]")
        assert np.abs(LSE[0, hi].cpu().numpy()[rows] - ref["LSE"]).max() <= P.LSE_MAX_ABS


def test_full_scope_refuses_kept_lists_and_noise():
    N = 256
    Q, K, V = (t.to(DEV) for t in synth.qkv(1, 1, N, 128))
    S = synth.scores(1, 1, N, 4).to(DEV)
    layer = sas.SasLayer(1, 1, N, 128, 2, scope=sas.SAS_SCOPE_FULL)
    O = torch.empty_like(Q)
    si = torch.empty(1, 1, N, 2, device=DEV, dtype=torch.int32)
    with pytest.raises(sas.SasError):
        sas.sas_attention_fwd(layer.h, Q, K, V, O, S, sel_idx=si)
    with pytest.raises(sas.SasError):
        sas.sas_attention_fwd_noisy(layer.h, Q, K, V, O, torch.zeros_like(S), scores=S)
    layer.close()


# ------------------------------------------------------------------ full*

def test_noisy_zero_noise_is_the_sparse_path():
    # given scores: s + 0 = s exactly, so every output is bit-identical.  The
    # learned selector ranks the raw products q~.K~ in the sparse path but forms
    # s = q~.K~ / sqrt(d_sel) before adding noise, so there the kept sets agree
    # and the log-gates and outputs agree to rounding.
    B, H, N, d, topk = 1, 2, 1000, 128, 4
    Q, K, V = (t.to(DEV) for t in synth.qkv(B, H, N, d, seed=8, regime="R2"))
    Wq, Wk = (t.to(DEV) for t in synth.selector_weights(H, d, d, seed=8))
    S = synth.scores(B, H, N, -(-N // 64), seed=8).to(DEV)
    zero = torch.zeros_like(S)
    for kw in (dict(scores=S), dict(Wq=Wq, Wk=Wk)):
        sel = sas.SAS_SEL_SCORES_GIVEN if "scores" in kw else sas.SAS_SEL_MEANPOOL_PROJ
        layer = sas.SasLayer(B, H, N, d, topk, selector=sel)
        a = layer.attention(Q, K, V, **kw)
        b = layer.attention_noisy(Q, K, V, zero, **kw)
        torch.cuda.synchronize()
        layer.close()
        if sel == sas.SAS_SEL_SCORES_GIVEN:
            for x, y in zip(a, b):
                assert torch.equal(x, y)
        else:
            assert torch.equal(a[2], b[2])                                   # kept sets
            assert float((a[3] - b[3]).abs().max()) <= 1e-5                  # log-gates
            assert float((a[0].float() - b[0].float()).abs().max()) <= 2e-2  # O
            assert float((a[1] - b[1]).abs().max()) <= 1e-4                  # LSE


def test_noisy_given_scores_match_oracle():
    # the scores and the noise are fp32, their sum is formed in fp32 on both
    # sides, so the kept sets are bit-exact
    B, H, N, d, topk = 1, 2, 1000, 128, 4
    Q, K, V = synth.qkv(B, H, N, d, seed=9)
    C = -(-N // 64)
    S = synth.scores(B, H, N, C, seed=9, regime="R1")
    E = synth.normal((B, H, N, C), seed=99, std=0.5)
    layer = sas.SasLayer(B, H, N, d, topk, selector=sas.SAS_SEL_SCORES_GIVEN)
    O, LSE, si, sl = layer.attention_noisy(Q.to(DEV), K.to(DEV), V.to(DEV), E.to(DEV), scores=S.to(DEV))
    torch.cuda.synchronize()
    layer.close()
    for hi in range(H):
        sn = OR.noisy_scores(P.f64(S[0, hi]), P.f64(E[0, hi]))
        ref = OR.sas_attention_head(P.f64(Q[0, hi]), P.f64(K[0, hi]), P.f64(V[0, hi]), sn, 64, topk)
        rr = np.arange(N)
        P.check_selection_rows(si[0, hi].cpu().numpy()[:, :topk], sn, rr, topk)
        assert np.abs(sl[0, hi].cpu().numpy()[:, :topk] - ref["sel_logg"]).max(initial=0) <= P.LOGG_MAX_ABS
        P.compare_o(P.f64(O[0, hi].cpu()), ref["O"], f"O[0,{hi}]")
        # the noise changed the selection somewhere (it is not a no-op)
        plain = OR.sas_attention_head(P.f64(Q[0, hi]), P.f64(K[0, hi]), P.f64(V[0, hi]), P.f64(S[0, hi]), 64, topk,
                                      rows=np.arange(512, N))
        assert not np.array_equal(plain["sel_idx"], ref["sel_idx"][512:])


def test_noisy_learned_selector_matches_oracle():
    # integer inputs make every product exact; the GPU forms s = fp32(u / sqrt(d_sel))
    # before adding the noise, which may sit one fp32 step from the oracle's sum:
    # rows whose K-th / (K+1)-th margin exceeds that must match exactly
    B, H, N, d, topk = 1, 2, 1200, 128, 5
    Q, K, V, Wq, Wk = synth.integer_selector_inputs(B, H, N, d, d, seed=10)
    C = -(-N // 64)
    E = synth.normal((B, H, N, C), seed=100, std=0.5)
    layer = sas.SasLayer(B, H, N, d, topk, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d)
    O, LSE, si, sl = layer.attention_noisy(Q.to(DEV), K.to(DEV), V.to(DEV), E.to(DEV), Wq=Wq.to(DEV), Wk=Wk.to(DEV))
    torch.cuda.synchronize()
    layer.close()
    rr = np.arange(N)
    for hi in range(H):
        s = P.oracle_scores(Q, K, Wq, Wk, 0, hi)   # [N, floor(N/64)]: blocks that can be historical
        sn = OR.noisy_scores(s, P.f64(E[0, hi])[:, :s.shape[1]])
        tol = np.full(N, 4 * 2.0 ** -23 * (np.abs(sn).max() + 1.0))
        _, _, mism = P.check_selection_rows(si[0, hi].cpu().numpy()[:, :topk], sn, rr, topk, tol)
        ref = OR.sas_attention_head(P.f64(Q[0, hi]), P.f64(K[0, hi]), P.f64(V[0, hi]), sn, 64, topk)
        keep = ~mism
        P.compare_o(P.f64(O[0, hi].cpu())[keep], ref["O"][keep], f"O[0,{hi}]")
        assert mism.sum() <= 0.01 * N
