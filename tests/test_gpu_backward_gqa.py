"""GPU parity of the SAS backward under grouped-query attention (Sec. 3.3:
the G query heads of a KV group share its K, V, kept blocks and gates)
against the fp64 oracle's sas_attention_bwd_gqa, through the C ABI.

dQ is per query head; dK, dV and d(log g) of a group are the sums of its
heads' contributions, and the score gradient applies the gate softmax's
Jacobian (App. D) to the summed d(log g)."""
import numpy as np
import pytest
import torch

from oracle import backward_oracle as BO
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu

TRAIN, INFER = sas.SAS_MODE_TRAIN_SOFT, sas.SAS_MODE_INFER_HARD
DEV = "cuda:0"


def _inputs(B, Hq, Hkv, N, seed):
    d = 128
    Q = synth.qkv(B, Hq, N, d, seed=seed)[0]
    _, K, V = synth.qkv(B, Hkv, N, d, seed=seed + 100)
    S = synth.scores(B, Hkv, N, -(-N // 64), seed=seed, regime="R1")
    dO = synth.normal((B, Hq, N, d), seed + 5).to(torch.bfloat16)
    return Q, K, V, S, dO


def _gpu(B, Hq, Hkv, N, topk, mode, Q, K, V, S, dO, want_ds=True):
    layer = sas.SasLayer(B, Hq, N, 128, topk, mode=mode, Hkv=Hkv)
    cu = lambda t: t.to(DEV).contiguous()
    Qd, Kd, Vd, Sd, dOd = cu(Q), cu(K), cu(V), cu(S), cu(dO)
    O, LSE, si, sl = layer.attention(Qd, Kd, Vd, scores=Sd)
    dQ, dK, dV, dlogg, ds = layer.attention_bwd(Qd, Kd, Vd, O, LSE, dOd, scores=Sd, sel_idx=si, sel_logg=sl,
                                                want_ds=want_ds)
    torch.cuda.synchronize()
    status = sas.sas_get_device_status(layer.h)
    layer.close()
    return {"O": O.cpu(), "dQ": dQ.cpu(), "dK": dK.cpu(), "dV": dV.cpu(), "dlogg": dlogg.cpu(),
            "ds": None if ds is None else ds.cpu(), "status": status}


def _check_group(g, Q, K, V, S, dO, bi, gk, G, topk, mode, rows=None, keys=None):
    """One KV group of batch element bi: the oracle's group backward against
    the GPU's, each bf16 gradient within its derived bound (the per-head
    bounds of P.grad_extra, summed over the group's heads for dK, dV)."""
    N = Q.shape[2]
    rows = np.arange(N) if rows is None else rows
    keys = np.arange(N) if keys is None else keys
    hs = range(gk * G, (gk + 1) * G)
    s = P.f64(S[bi, gk])
    ref = BO.sas_attention_bwd_gqa(P.f64(Q[bi, gk * G:(gk + 1) * G]), P.f64(K[bi, gk:gk + 1]),
                                   P.f64(V[bi, gk:gk + 1]), s[None], P.f64(dO[bi, gk * G:(gk + 1) * G]), 64, topk,
                                   mode)
    ek = np.zeros((N, 128))
    ev = np.zeros((N, 128))
    tol = np.zeros(N)
    for j, h in enumerate(hs):
        ex = P.grad_extra(P.f64(Q[bi, h]), P.f64(K[bi, gk]), P.f64(V[bi, gk]), s, P.f64(dO[bi, h]),
                          P.f64(g["O"][bi, h]), 64, topk, mode)
        P.compare_o(P.f64(g["dQ"][bi, h])[rows], ref["dQ"][j][rows], f"dQ[{bi},{h}]", ex["dQ"][rows])
        ek += ex["dK"]
        ev += ex["dV"]
        tol += 2.0 ** -8 * np.abs(P.f64(g["O"][bi, h]) * P.f64(dO[bi, h])).sum(axis=-1) + 1e-4
    P.compare_o(P.f64(g["dK"][bi, gk])[keys], ref["dK"][0][keys], f"dK[{bi},{gk}]", ek[keys])
    P.compare_o(P.f64(g["dV"][bi, gk])[keys], ref["dV"][0][keys], f"dV[{bi},{gk}]", ev[keys])
    if topk > 0:
        gl = g["dlogg"][bi, gk].numpy()[rows][:, :topk]
        assert np.all(np.abs(gl - ref["dlogg"][0][rows]) <= tol[rows][:, None]), "dlogg"
    if g["ds"] is not None:
        gds = g["ds"][bi, gk].numpy()[rows]
        assert np.all(np.abs(gds - ref["ds"][0][rows]) <= 2 * tol[rows][:, None]), "ds"


@pytest.mark.parametrize("B,Hq,Hkv,N,topk,mode", [
    (1, 8, 2, 700, 4, TRAIN),     # G = 4, ragged tail, several tiles
    (2, 6, 3, 389, 2, TRAIN),     # G = 2, two batch elements
    (1, 4, 1, 517, 3, TRAIN),     # MQA: one KV head for all four query heads
    (1, 4, 2, 600, 3, INFER),     # inference form: no gate gradient
])
def test_gqa_backward_matches_oracle(B, Hq, Hkv, N, topk, mode):
    Q, K, V, S, dO = _inputs(B, Hq, Hkv, N, seed=Hq + N)
    g = _gpu(B, Hq, Hkv, N, topk, mode, Q, K, V, S, dO)
    assert g["status"] == 0
    G = Hq // Hkv
    for bi in range(B):
        for gk in range(Hkv):
            _check_group(g, Q, K, V, S, dO, bi, gk, G, topk, mode)
    if mode == INFER:
        assert float(g["dlogg"][..., :topk].abs().max()) == 0.0
        assert float(g["ds"].abs().max()) == 0.0


def test_gqa_backward_against_mha_on_repeated_inputs():
    # The MHA backward on per-head copies of K, V and the scores runs the same
    # pass 1 per query head: dQ is bit-identical, and the group's d(log g) is
    # the fp32 sum, in head order, of the MHA heads' (bit-identical).  dK, dV
    # are sums of the same products accumulated across the group's heads in
    # one fp32 accumulator, so they match the sum of the MHA heads' within
    # the bf16 rounding of each term.
    B, Hq, Hkv, N, topk = 1, 8, 2, 900, 4
    G = Hq // Hkv
    Q, K, V, S, dO = _inputs(B, Hq, Hkv, N, seed=11)
    g = _gpu(B, Hq, Hkv, N, topk, TRAIN, Q, K, V, S, dO, want_ds=False)
    rep = lambda t: t.repeat_interleave(G, dim=1)
    m = _gpu(B, Hq, Hq, N, topk, TRAIN, Q, rep(K), rep(V), rep(S), dO, want_ds=False)
    assert g["status"] == 0 and m["status"] == 0
    assert torch.equal(g["O"], m["O"])
    assert torch.equal(g["dQ"], m["dQ"])
    per_head = m["dlogg"].numpy().astype(np.float32).reshape(B, Hkv, G, N, -1)
    acc = np.zeros_like(per_head[:, :, 0])
    for j in range(G):
        acc = (acc + per_head[:, :, j]).astype(np.float32)
    assert np.array_equal(g["dlogg"].numpy(), acc)
    for name in ("dK", "dV"):
        heads = P.f64(m[name]).reshape(B, Hkv, G, N, 128)
        want = heads.sum(axis=2)
        # per-term bf16 roundings, plus the fp32 accumulation order (a floor of
        # 2^-10 of the largest value, far below a missing or doubled head)
        bound = 2.0 ** -8 * np.abs(heads).sum(axis=2) + 2.0 ** -8 * np.abs(want) + 2.0 ** -10 * np.abs(want).max()
        assert np.all(np.abs(P.f64(g[name]) - want) <= bound), name


def test_gqa_backward_repeated_calls_identical():
    B, Hq, Hkv, N, topk = 1, 8, 2, 800, 4
    Q, K, V, S, dO = _inputs(B, Hq, Hkv, N, seed=12)
    a = _gpu(B, Hq, Hkv, N, topk, TRAIN, Q, K, V, S, dO)
    b = _gpu(B, Hq, Hkv, N, topk, TRAIN, Q, K, V, S, dO)
    for k in ("dQ", "dK", "dV", "dlogg", "ds"):
        assert torch.equal(a[k], b[k]), k


def test_qwen3_4b_shaped_gqa_backward_sampled():
    # Hq = 32, Hkv = 8 (G = 4), d = 128, K = 32 at 4096 tokens: two groups
    # checked on sampled rows (dQ, dlogg, ds) and sampled keys (dK, dV)
    B, Hq, Hkv, N, topk = 1, 32, 8, 4096, 32
    Q, K, V, S, dO = _inputs(B, Hq, Hkv, N, seed=13)
    g = _gpu(B, Hq, Hkv, N, topk, TRAIN, Q, K, V, S, dO)
    assert g["status"] == 0
    rows = P.sample_rows(N, n_random=96, seed=2)
    for gk in (0, 7):
        _check_group(g, Q, K, V, S, dO, 0, gk, 4, topk, TRAIN, rows=rows, keys=rows)
