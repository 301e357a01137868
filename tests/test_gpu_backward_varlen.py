"""GPU parity of the SAS backward over packed variable-length sequences (each
sequence its own causal problem with its own block partition; no gradient
crosses sequences) against the fp64 oracle's sas_attention_bwd_varlen,
bit-identity with the batched backward on equal lengths, and rows past the
last sequence left unwritten."""
import numpy as np
import pytest
import torch

from oracle import backward_oracle as BO
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu

TRAIN, INFER = sas.SAS_MODE_TRAIN_SOFT, sas.SAS_MODE_INFER_HARD
DEV = torch.device("cuda:0")


def _packed(lens, cap, Hq, Hkv, max_len, seed):
    d = 128
    Q = synth.qkv(1, Hq, cap, d, seed=seed)[0][0]
    _, K, V = synth.qkv(1, Hkv, cap, d, seed=seed + 100)
    S = synth.scores(1, Hkv, cap, -(-max_len // 64), seed=seed, regime="R1")[0]
    dO = synth.normal((Hq, cap, d), seed + 5).to(torch.bfloat16)
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32)
    return Q, K[0], V[0], S, dO, cu


def _run(lens, cap, Hq, Hkv, topk, mode, max_len, Q, K, V, S, dO, cu, want_ds=True):
    layer = sas.SasLayer(1, Hq, cap, 128, topk, mode=mode, Hkv=Hkv, max_seqs=max(len(lens), 1), max_seqlen=max_len)
    d = lambda t: t.to(DEV).contiguous()
    Qd, Kd, Vd, Sd, dOd = d(Q), d(K), d(V), d(S), d(dO)
    O, LSE, si, sl = layer.attention_varlen(d(cu), Qd, Kd, Vd, Sd)
    dQ, dK, dV, dlogg, ds = layer.attention_bwd_varlen(Qd, Kd, Vd, O, LSE, dOd, scores=Sd, sel_idx=si, sel_logg=sl,
                                                       want_ds=want_ds)
    torch.cuda.synchronize()
    status = sas.sas_get_device_status(layer.h)
    layer.close()
    return {"O": O.cpu(), "dQ": dQ.cpu(), "dK": dK.cpu(), "dV": dV.cpu(), "dlogg": dlogg.cpu(),
            "ds": None if ds is None else ds.cpu(), "status": status}


def _check(g, Q, K, V, S, dO, cu, topk, mode, groups=None, rows=None):
    """Every sequence of the listed KV groups against the oracle, each bf16
    gradient within the derived bounds of P.grad_extra on the sequence's slice
    (summed over a group's heads for dK, dV; rows = sampled token positions)."""
    Hq, Hkv = Q.shape[0], K.shape[0]
    G = Hq // Hkv
    cu = [int(x) for x in cu]
    ref = BO.sas_attention_bwd_varlen(P.f64(Q), P.f64(K), P.f64(V), P.f64(S), P.f64(dO), cu, 64, topk, mode)
    want = set(range(cu[-1])) if rows is None else set(int(r) for r in rows)
    for gk in (range(Hkv) if groups is None else groups):
        for s0, s1 in zip(cu[:-1], cu[1:]):
            sel = np.array(sorted(r - s0 for r in want if s0 <= r < s1), dtype=np.int64)
            if s1 == s0 or sel.size == 0:
                continue
            sl = slice(s0, s1)
            s = P.f64(S[gk, sl])
            ek = np.zeros((s1 - s0, 128))
            ev = np.zeros((s1 - s0, 128))
            tol = np.zeros(s1 - s0)
            for h in range(gk * G, (gk + 1) * G):
                ex = P.grad_extra(P.f64(Q[h, sl]), P.f64(K[gk, sl]), P.f64(V[gk, sl]), s, P.f64(dO[h, sl]),
                                  P.f64(g["O"][h, sl]), 64, topk, mode)
                P.compare_o(P.f64(g["dQ"][h, sl])[sel], ref["dQ"][h, sl][sel], f"dQ[{h}, seq@{s0}]", ex["dQ"][sel])
                ek += ex["dK"]
                ev += ex["dV"]
                tol += 2.0 ** -8 * np.abs(P.f64(g["O"][h, sl]) * P.f64(dO[h, sl])).sum(axis=-1) + 1e-4
            P.compare_o(P.f64(g["dK"][gk, sl])[sel], ref["dK"][gk, sl][sel], f"dK[{gk}, seq@{s0}]", ek[sel])
            P.compare_o(P.f64(g["dV"][gk, sl])[sel], ref["dV"][gk, sl][sel], f"dV[{gk}, seq@{s0}]", ev[sel])
            if topk > 0:
                gl = g["dlogg"][gk, sl].numpy()[sel][:, :topk]
                assert np.all(np.abs(gl - ref["dlogg"][gk, sl][sel]) <= tol[sel][:, None]), "dlogg"
            if g["ds"] is not None:
                Cs = ref["ds"].shape[2]
                gds = g["ds"][gk, sl].numpy()[sel][:, :Cs]
                assert np.all(np.abs(gds - ref["ds"][gk, sl][sel]) <= 2 * tol[sel][:, None]), "ds"
                assert float(np.abs(g["ds"][gk, sl].numpy()[:, Cs:]).max(initial=0.0)) == 0.0


def _untouched_past_end(g, end):
    for k in ("dQ", "dK", "dV", "dlogg", "ds"):
        if g[k] is not None:
            assert torch.count_nonzero(g[k][:, end:]) == 0, k


@pytest.mark.parametrize("lens,cap,Hq,Hkv,topk,mode", [
    ([700, 1, 64, 129, 0, 300, 255], 1500, 4, 2, 3, TRAIN),   # ragged, empty, one-token, GQA, spare rows
    ([513, 130, 77], 720, 2, 2, 2, TRAIN),                     # offsets off the block grid
    ([400, 250], 700, 2, 1, 2, INFER),                         # MQA, inference form: no gate gradient
    ([300, 129, 64, 1, 190], 700, 8, 1, 3, TRAIN),             # G = 8: head-packed tiles of 16 tokens, empty ones
])
def test_packed_backward_matches_oracle(lens, cap, Hq, Hkv, topk, mode):
    max_len = max(lens)
    Q, K, V, S, dO, cu = _packed(lens, cap, Hq, Hkv, max_len, seed=len(lens) + cap)
    g = _run(lens, cap, Hq, Hkv, topk, mode, max_len, Q, K, V, S, dO, cu)
    assert g["status"] == 0
    _check(g, Q, K, V, S, dO, cu.numpy(), topk, mode)
    _untouched_past_end(g, int(cu[-1]))
    if mode == INFER:
        assert float(g["dlogg"].abs().max()) == 0.0
        assert float(g["ds"].abs().max()) == 0.0


@pytest.mark.parametrize("H,Hkv", [(4, 4), (8, 2)])   # per-head tiles; head-packed tiles of 32 tokens x 4 heads
def test_packed_backward_equal_lengths_bit_identical_to_batched(H, Hkv):
    # Same data as a [B = 3, H, n, d] batch: pass 1 runs the same tiles, and pass
    # 2 sums a key pair's query tiles in the same order (by index within the
    # sequence), so every gradient is bit-identical.
    S_, n, topk = 3, 700, 4
    Q, K, V, S, dO, cu = _packed([n] * S_, S_ * n, H, Hkv, n, seed=9)
    g = _run([n] * S_, S_ * n, H, Hkv, topk, TRAIN, n, Q, K, V, S, dO, cu)
    assert g["status"] == 0
    bat = lambda x: x.reshape(x.shape[0], S_, n, -1).transpose(0, 1).contiguous().to(DEV)
    layer = sas.SasLayer(S_, H, n, 128, topk, Hkv=Hkv)
    Qb, Kb, Vb, Sb, dOb = bat(Q), bat(K), bat(V), bat(S), bat(dO)
    O, LSE, si, sl = layer.attention(Qb, Kb, Vb, scores=Sb)
    out = layer.attention_bwd(Qb, Kb, Vb, O, LSE, dOb, scores=Sb, sel_idx=si, sel_logg=sl, want_ds=True)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    unb = lambda x: x.cpu().transpose(0, 1).reshape(x.shape[1], S_ * n, -1)
    for k, b in zip(("dQ", "dK", "dV", "dlogg", "ds"), out):
        assert torch.equal(g[k], unb(b)), k


def test_long_gqa_pack_backward_sampled():
    lens = [3000, 64, 2100, 1]
    cap, Hq, Hkv, topk = 6000, 8, 2, 16
    Q, K, V, S, dO, cu = _packed(lens, cap, Hq, Hkv, 3000, seed=21)
    g = _run(lens, cap, Hq, Hkv, topk, TRAIN, 3000, Q, K, V, S, dO, cu)
    assert g["status"] == 0
    rows = P.sample_rows(int(cu[-1]), n_random=128, seed=3)
    _check(g, Q, K, V, S, dO, cu.numpy(), topk, TRAIN, groups=[1], rows=rows)
    _untouched_past_end(g, int(cu[-1]))
