"""GPU parity of the two backwards that gate every historical block, against
the fp64 oracle, through the C ABI:

* the full training scope (Sec. 4.2, Eq. scope_grad): every historical block
  kept and gated; oracle = the sparse backward keeping all blocks;
* the hard Top-K gate under the straight-through estimator (Sec. 4.2 ranking
  preservation, App. D, Eq. rank_unbounded): dQ, dK, dV of the hard forward,
  the gate gradient of every historical block (dropped ones included) and its
  score gradient; oracle = sas_attention_bwd_ste_gqa.

Tolerances: dQ, dK, dV use the derived bounds of parity.grad_extra (summed
over a group's heads).  dlogg (per block) and ds: Delta = dO . O uses the
forward's bf16 O, so it may sit dDelta = 2^-8 sum |dO O| from the exact
value; a block's entry moves by its probability mass times dDelta (the mass
of a dropped block under the hard normaliser can exceed 1, Eq.
rank_unbounded, so the mass is computed here), ds by twice the row's total,
plus 1e-4 for the fp32 sums."""
import math

import numpy as np
import pytest
import torch

from oracle import backward_oracle as BO
from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu

TRAIN, INFER, STE = sas.SAS_MODE_TRAIN_SOFT, sas.SAS_MODE_INFER_HARD, sas.SAS_MODE_TRAIN_HARD_STE
DEV = "cuda:0"


def _inputs(H, Hkv, N, seed):
    d = 128
    C = -(-N // 64)
    Q = synth.qkv(1, H, N, d, seed=seed)[0]
    _, K, V = synth.qkv(1, Hkv, N, d, seed=seed + 50)
    S = synth.scores(1, Hkv, N, C, seed=seed, regime="R1")
    dO = synth.normal((1, H, N, d), seed + 5).to(torch.bfloat16)
    return Q, K, V, S, dO


def _run(layer, Q, K, V, S, dO):
    d = lambda t: t.to(DEV).contiguous()
    Qd, Kd, Vd, Sd, dOd = d(Q), d(K), d(V), d(S), d(dO)
    O, LSE, si, sl = layer.attention(Qd, Kd, Vd, scores=Sd)
    out = layer.attention_bwd(Qd, Kd, Vd, O, LSE, dOd, scores=Sd, sel_idx=si, sel_logg=sl, want_ds=True)
    torch.cuda.synchronize()
    status = sas.sas_get_device_status(layer.h)
    layer.close()
    g = dict(zip(("dQ", "dK", "dV", "dlogg", "ds"), (t.cpu() for t in out)))
    g["O"] = O.cpu()
    g["status"] = status
    return g


def _check_qkv(g, Q, K, V, S, dO, topk, mode, rows=None, act=sas.SAS_GATE_SOFTMAX, pos=sas.SAS_GATE_INNER):
    """dQ per head, dK and dV per group, each within the summed derived bounds."""
    H, Hkv = Q.shape[1], K.shape[1]
    G = H // Hkv
    N = Q.shape[2]
    rr = np.arange(N) if rows is None else rows
    ref = BO.sas_attention_bwd_gqa(P.f64(Q[0]), P.f64(K[0]), P.f64(V[0]), P.f64(S[0]), P.f64(dO[0]), 64, topk, mode,
                                   act=act, pos=pos)
    for gk in range(Hkv):
        ek = np.zeros((N, 128))
        ev = np.zeros((N, 128))
        for h in range(gk * G, (gk + 1) * G):
            ex = P.grad_extra(P.f64(Q[0, h]), P.f64(K[0, gk]), P.f64(V[0, gk]), P.f64(S[0, gk]), P.f64(dO[0, h]),
                              P.f64(g["O"][0, h]), 64, topk, mode, act=act, pos=pos)
            P.compare_o(P.f64(g["dQ"][0, h])[rr], ref["dQ"][h][rr], f"dQ[{h}]", ex["dQ"][rr])
            ek += ex["dK"]
            ev += ex["dV"]
        P.compare_o(P.f64(g["dK"][0, gk])[rr], ref["dK"][gk][rr], f"dK[{gk}]", ek[rr])
        P.compare_o(P.f64(g["dV"][0, gk])[rr], ref["dV"][gk][rr], f"dV[{gk}]", ev[rr])
    return ref


def _delta_err(O, dO):
    return 2.0 ** -8 * np.abs(P.f64(O) * P.f64(dO)).sum(axis=-1)


def _block_mass(Q, K, LSE_ref, i, c, sm_scale):
    """Probability mass of each historical block of row i under the normaliser LSE_ref."""
    z = sm_scale * (K[:c * 64] @ Q[i]) - LSE_ref
    return np.exp(z).reshape(c, 64).sum(axis=1)


# ------------------------------------------------------------------ full scope

@pytest.mark.parametrize("H,Hkv,N,mode,seed", [
    (2, 2, 700, TRAIN, 1),     # ragged, several tiles
    (4, 2, 517, TRAIN, 2),     # GQA: dK, dV and the gate gradients summed over the group
    (2, 2, 600, INFER, 3),     # dense causal attention, no gate gradient
])
def test_full_scope_backward_matches_oracle(H, Hkv, N, mode, seed):
    Q, K, V, S, dO = _inputs(H, Hkv, N, seed)
    C = -(-N // 64)
    layer = sas.SasLayer(1, H, N, 128, 4, mode=mode, Hkv=Hkv, scope=sas.SAS_SCOPE_FULL)
    g = _run(layer, Q, K, V, S, dO)
    assert g["status"] == 0
    assert g["dlogg"].shape == (1, Hkv, N, C)
    ref = _check_qkv(g, Q, K, V, S, dO, C, mode)
    G = H // Hkv
    for gk in range(Hkv):
        tol = sum(_delta_err(g["O"][0, h], dO[0, h]) for h in range(gk * G, (gk + 1) * G)) + 1e-4
        gl = g["dlogg"][0, gk].numpy()
        for i in range(N):
            c = i // 64
            assert np.all(np.abs(gl[i, :c] - ref["dlogg"][gk, i, :c]) <= tol[i]), ("dlogg", gk, i)
        gds = g["ds"][0, gk].numpy()
        assert np.all(np.abs(gds - ref["ds"][gk]) <= 2 * tol[:, None]), "ds"
    if mode == INFER:
        assert float(g["dlogg"].abs().max()) == 0.0 and float(g["ds"].abs().max()) == 0.0


def test_full_scope_backward_beyond_64_blocks():
    # N = 4608: rows past token 4096 keep and gate 65 .. 71 historical blocks,
    # more than any Top-K the sparse scope allows
    N = 4608
    Q, K, V, S, dO = _inputs(1, 1, N, 7)
    layer = sas.SasLayer(1, 1, N, 128, 4, Hkv=1, scope=sas.SAS_SCOPE_FULL)
    g = _run(layer, Q, K, V, S, dO)
    assert g["status"] == 0
    rows = P.sample_rows(N, n_random=96, seed=4)
    rows = np.unique(np.concatenate([rows, np.arange(N - 64, N)]))
    C = -(-N // 64)
    ref = _check_qkv(g, Q, K, V, S, dO, C, TRAIN, rows=rows)
    tol = _delta_err(g["O"][0, 0], dO[0, 0]) + 1e-4
    gl = g["dlogg"][0, 0].numpy()
    for i in rows:
        c = i // 64
        assert np.all(np.abs(gl[i, :c] - ref["dlogg"][0, i, :c]) <= tol[i])
    assert np.all(np.abs(g["ds"][0, 0].numpy()[rows] - ref["ds"][0][rows]) <= 2 * tol[rows][:, None])


# ----------------------------------------------------- hard gate with STE

@pytest.mark.parametrize("H,Hkv,N,topk,seed", [
    (2, 2, 700, 3, 11),        # ragged, several tiles
    (4, 2, 517, 2, 12),        # GQA (head-packed tiles in the hard backward)
    (2, 2, 300, 0, 13),        # K = 0: every historical block is dropped
    (2, 2, 250, 8, 14),        # K >= C_i: every historical block is kept (the gates are all 1)
])
def test_ste_backward_matches_oracle(H, Hkv, N, topk, seed):
    Q, K, V, S, dO = _inputs(H, Hkv, N, seed)
    layer = sas.SasLayer(1, H, N, 128, topk, mode=STE, Hkv=Hkv)
    g = _run(layer, Q, K, V, S, dO)
    assert g["status"] == 0
    # the forward is the hard one, bit for bit
    hard = sas.SasLayer(1, H, N, 128, topk, mode=INFER, Hkv=Hkv)
    Oh, _, _, _ = hard.attention(Q.to(DEV), K.to(DEV), V.to(DEV), scores=S.to(DEV))
    torch.cuda.synchronize()
    hard.close()
    assert torch.equal(g["O"], Oh.cpu())
    _check_qkv(g, Q, K, V, S, dO, topk, INFER)
    ref = BO.sas_attention_bwd_ste_gqa(P.f64(Q[0]), P.f64(K[0]), P.f64(V[0]), P.f64(S[0]), P.f64(dO[0]), 64, topk)
    G = H // Hkv
    sm = 1 / math.sqrt(128)
    for gk in range(Hkv):
        gx = g["dlogg"][0, gk].numpy()
        gds = g["ds"][0, gk].numpy()
        for i in range(64, N, 7):
            c = i // 64
            gates = np.exp(OR.log_gates(P.f64(S[0, gk, i, :c])))
            tol = np.full(c, 1e-4)
            for h in range(gk * G, (gk + 1) * G):
                fwd = OR.sas_attention_head(P.f64(Q[0, h]), P.f64(K[0, gk]), P.f64(V[0, gk]), P.f64(S[0, gk]), 64,
                                            topk, INFER, rows=[i])
                mass = _block_mass(P.f64(Q[0, h]), P.f64(K[0, gk]), fwd["LSE"][0], i, c, sm)
                tol += gates * np.maximum(mass, 1e-30) * _delta_err(g["O"][0, h, i], dO[0, h, i]) * 2
                tol += gates * mass * 1e-3   # fp32 logits and exp2 of the kernel
            tol += 1e-5 * np.abs(ref["x"][gk, i, :c])
            assert np.all(np.abs(gx[i, :c] - ref["x"][gk, i, :c]) <= tol), ("x", gk, i)
            assert np.all(np.abs(gds[i, :c] - ref["ds"][gk, i, :c]) <= 2 * tol.sum()), ("ds", gk, i)
            assert np.all(gx[i, c:] == 0) and np.all(gds[i, c:] == 0)


def test_ste_rejects_what_it_does_not_cover():
    # the estimator needs the soft gates of every block: given scores, sparse scope, softmax inner
    with pytest.raises(sas.SasError):
        sas.SasLayer(1, 2, 256, 128, 2, mode=STE, scope=sas.SAS_SCOPE_FULL)
    with pytest.raises(sas.SasError):
        sas.SasLayer(1, 2, 256, 128, 2, mode=STE, gate_act=sas.SAS_GATE_SIGMOID)
    # packed sequences: the forward runs, the estimator's backward is refused before any launch
    N, d = 512, 128
    layer = sas.SasLayer(1, 2, N, d, 2, mode=STE, max_seqs=2, max_seqlen=300)
    Q, K, V = (t[0].to(DEV) for t in synth.qkv(1, 2, N, d, seed=3))
    S = synth.scores(1, 2, N, 5, seed=3)[0].to(DEV)
    cu = torch.tensor([0, 300, 512], dtype=torch.int32, device=DEV)
    O, LSE, si, sl = layer.attention_varlen(cu, Q, K, V, S)
    with pytest.raises(sas.SasError, match="take \\[B, H, N, d\\] inputs"):
        layer.attention_bwd_varlen(Q, K, V, O, LSE, torch.zeros_like(Q), scores=S, sel_idx=si, sel_logg=sl)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()


# --------------------------------------------------------------------- full*

def test_noisy_scope_backward_is_the_sparse_backward_at_the_noisy_scores():
    # full* (Table 1 setting 11): s~ = s + eps chooses and gates the blocks, and
    # ds = ds~, so the backward is the sparse one evaluated at s~ (passed as the
    # scores); the oracle runs on fp32(s + eps)
    H, N, topk = 2, 700, 3
    Q, K, V, S, dO = _inputs(H, H, N, 21)
    eps = (0.5 * synth.normal(tuple(S.shape), 77)).to(torch.float32)
    St = (S + eps).to(torch.float32)                         # the fp32 sum the forward forms
    d = lambda t: t.to(DEV).contiguous()
    layer = sas.SasLayer(1, H, N, 128, topk)
    Qd, Kd, Vd, dOd = d(Q), d(K), d(V), d(dO)
    O, LSE, si, sl = layer.attention_noisy(Qd, Kd, Vd, d(eps), scores=d(S))
    out = layer.attention_bwd(Qd, Kd, Vd, O, LSE, dOd, scores=d(St), sel_idx=si, sel_logg=sl, want_ds=True)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    g = dict(zip(("dQ", "dK", "dV", "dlogg", "ds"), (t.cpu() for t in out)))
    g["O"] = O.cpu()
    s_noisy = OR.noisy_scores(P.f64(S), P.f64(eps))
    ref = _check_qkv(g, Q, K, V, torch.from_numpy(s_noisy), dO, topk, TRAIN)
    for h in range(H):
        tol = _delta_err(g["O"][0, h], dO[0, h]) + 1e-4
        gl = g["dlogg"][0, h].numpy()[:, :topk]
        assert np.all(np.abs(gl - ref["dlogg"][h]) <= tol[:, None]), "dlogg"
        assert np.all(np.abs(g["ds"][0, h].numpy() - ref["ds"][h]) <= 2 * tol[:, None]), "ds"


# ------------------------------------------------ outer gate position, GQA

def test_outer_gate_position_gqa_backward():
    # o = softmax(z) (g . V) under GQA (head-packed tiles in both passes): dK, dV
    # and the group's d(log g) are sums over its heads; ds from the summed dlogg
    H, Hkv, N, topk = 4, 2, 517, 2
    Q, K, V, S, dO = _inputs(H, Hkv, N, 31)
    layer = sas.SasLayer(1, H, N, 128, topk, Hkv=Hkv, gate_pos=sas.SAS_GATE_OUTER)
    g = _run(layer, Q, K, V, S, dO)
    assert g["status"] == 0
    ref = _check_qkv(g, Q, K, V, S, dO, topk, TRAIN, pos=sas.SAS_GATE_OUTER)
    G = H // Hkv
    for gk in range(Hkv):
        tol = sum(_delta_err(g["O"][0, h], dO[0, h]) for h in range(gk * G, (gk + 1) * G)) + 1e-4
        gl = g["dlogg"][0, gk].numpy()[:, :topk]
        assert np.all(np.abs(gl - ref["dlogg"][gk]) <= tol[:, None]), "dlogg"
        assert np.all(np.abs(g["ds"][0, gk].numpy() - ref["ds"][gk]) <= 2 * tol[:, None]), "ds"


def test_full_scope_backward_learned_selector():
    # the learned selector's full scope: the handle's score table supplies the
    # log-gates of every block (integer Q, K and sparse {-1, 0, 1} projections,
    # so the kernel's scores are exact and equal the oracle's)
    B, H, N, d = 1, 2, 900, 128
    Q, K, V, Wq, Wk = synth.integer_selector_inputs(B, H, N, d, d, seed=8)
    dO = synth.normal((B, H, N, d), 13).to(torch.bfloat16)
    dv = lambda t: t.to(DEV).contiguous()
    layer = sas.SasLayer(B, H, N, d, 4, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d, scope=sas.SAS_SCOPE_FULL)
    Qd, Kd, Vd, dOd = dv(Q), dv(K), dv(V), dv(dO)
    O, LSE, _, _ = layer.attention(Qd, Kd, Vd, Wq=dv(Wq), Wk=dv(Wk))
    dQ, dK, dV, dlogg, ds = layer.attention_bwd(Qd, Kd, Vd, O, LSE, dOd)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    C = -(-N // 64)
    assert ds is None and dlogg.shape == (B, H, N, C)
    for hi in range(H):
        s = P.oracle_scores(Q, K, Wq, Wk, 0, hi)
        args = (P.f64(Q[0, hi]), P.f64(K[0, hi]), P.f64(V[0, hi]), s, P.f64(dO[0, hi]))
        ref = BO.sas_attention_bwd_full_head(*args, 64)
        ex = P.grad_extra(*args, P.f64(O[0, hi].cpu()), 64, C, TRAIN)
        for name, gt in (("dQ", dQ), ("dK", dK), ("dV", dV)):
            P.compare_o(P.f64(gt[0, hi].cpu()), ref[name], f"{name}[{hi}]", ex[name])
        tol = _delta_err(O[0, hi].cpu(), dO[0, hi]) + 1e-4
        gl = dlogg[0, hi].cpu().numpy()
        for i in range(N):
            c = i // 64
            assert np.all(np.abs(gl[i, :c] - ref["dlogg"][i, :c]) <= tol[i]), ("dlogg", hi, i)
