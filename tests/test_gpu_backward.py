"""GPU parity of the SAS backward (Alg. 4; App. D gate and score gradients)
against the fp64 backward oracle, through the C ABI.  The forward runs on the
GPU first (its O, LSE and kept lists feed the backward, as in training)."""
import numpy as np
import pytest
import torch

from oracle import backward_oracle as BO
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu

TRAIN, INFER = sas.SAS_MODE_TRAIN_SOFT, sas.SAS_MODE_INFER_HARD
DEV = "cuda:0"
# dlogg and ds: Delta = dO . O uses the forward's bf16 O (Alg. 4), so Delta may
# sit up to 2^-8 sum_c |dO_c O_c| from the oracle's exact value; a block's
# dlogg moves by at most its probability mass (<= 1) times that, ds by twice it.
# Plus 1e-4 for the fp32 sums.
def _delta_bound(O, dO):
    return 2.0 ** -8 * np.abs(P.f64(O) * P.f64(dO)).sum(axis=-1) + 1e-4


def run_bwd(B, H, N, topk, mode, seed, learned=False, heads=None, rows=None, act=sas.SAS_GATE_SOFTMAX,
            pos=sas.SAS_GATE_INNER):
    d = 128
    C = -(-N // 64)
    if learned:
        Q, K, V = synth.qkv(B, H, N, d, seed=seed, regime="R2")
        Wq, Wk = synth.selector_weights(H, d, d, seed=seed)
        S = None
        layer = sas.SasLayer(B, H, N, d, topk, mode=mode, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d)
    else:
        Q, K, V = synth.qkv(B, H, N, d, seed=seed)
        S = synth.scores(B, H, N, C, seed=seed, regime="R1")
        layer = sas.SasLayer(B, H, N, d, topk, mode=mode, selector=sas.SAS_SEL_SCORES_GIVEN, gate_act=act,
                             gate_pos=pos)
    dO = synth.normal((B, H, N, d), seed + 5).to(torch.bfloat16)
    cu = lambda t: None if t is None else t.to(DEV).contiguous()
    Qd, Kd, Vd, dOd = cu(Q), cu(K), cu(V), cu(dO)
    if learned:
        O, LSE, si, sl = layer.attention(Qd, Kd, Vd, Wq=cu(Wq), Wk=cu(Wk))
    else:
        O, LSE, si, sl = layer.attention(Qd, Kd, Vd, scores=cu(S))
    dQ, dK, dV, dlogg, ds = layer.attention_bwd(Qd, Kd, Vd, O, LSE, dOd, scores=None if learned else cu(S),
                                                sel_idx=si, sel_logg=sl, want_ds=not learned)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    heads = heads or [(bi, hi) for bi in range(B) for hi in range(H)]
    for bi, hi in heads:
        if learned:
            s = P.oracle_scores(Q, K, Wq, Wk, bi, hi)
        else:
            s = P.f64(S[bi, hi])
        ref = BO.sas_attention_bwd_head(P.f64(Q[bi, hi]), P.f64(K[bi, hi]), P.f64(V[bi, hi]), s,
                                        P.f64(dO[bi, hi]), 64, topk, mode, act=act, pos=pos)
        rr = np.arange(N) if rows is None else rows
        extra = P.grad_extra(P.f64(Q[bi, hi]), P.f64(K[bi, hi]), P.f64(V[bi, hi]), s, P.f64(dO[bi, hi]),
                             P.f64(O[bi, hi].cpu()), 64, topk, mode, act=act, pos=pos)
        for name, g in (("dQ", dQ), ("dK", dK), ("dV", dV)):
            r = ref[name][rr]
            P.compare_o(P.f64(g[bi, hi].cpu())[rr], r, f"{name}[{bi},{hi}]", extra[name][rr])
        tol = _delta_bound(O[bi, hi].cpu(), dO[bi, hi])[rr][:, None]
        if topk > 0:
            gl = dlogg[bi, hi].cpu().numpy()[rr][:, :topk]
            assert np.all(np.abs(gl - ref["dlogg"][rr]) <= tol), "dlogg"
        if ds is not None:
            gds = ds[bi, hi].cpu().numpy()[rr]
            assert np.all(np.abs(gds - ref["ds"][rr]) <= 2 * tol), "ds"
    return dQ, dK, dV, dlogg, ds


def test_backward_ragged_multi_tile_train():
    # 1000 = 15 * 64 + 40: eight 128-row tiles, a partial last block
    run_bwd(1, 2, 1000, 4, TRAIN, seed=1)


@pytest.mark.parametrize("act", [sas.SAS_GATE_SIGMOID, sas.SAS_GATE_LOGIT])
def test_backward_other_gate_activations(act):
    # Sec. 4.2 gate activation: the same passes on the forward's log-gates; the
    # score gradient reaches kept blocks only (sigmoid: dlogg (1 - g), raw logit: dlogg)
    run_bwd(1, 2, 700, 3, TRAIN, seed=15, act=act)


@pytest.mark.parametrize("act", [sas.SAS_GATE_SOFTMAX, sas.SAS_GATE_SIGMOID])
def test_backward_outer_gate_position(act):
    # Sec. 4.2 gate position: o = softmax(z) (g . V); dV takes P g dO,
    # dS = P (g dP - Delta), a block's dlogg is the row sum of P g dP
    run_bwd(1, 2, 700, 3, TRAIN, seed=16, act=act, pos=sas.SAS_GATE_OUTER)


def test_backward_inference_mode_has_no_gate_gradient():
    _, _, _, dlogg, ds = run_bwd(1, 2, 700, 3, INFER, seed=2)
    assert float(dlogg[..., :3].abs().max()) == 0.0
    assert float(ds.abs().max()) == 0.0


@pytest.mark.parametrize("N,topk", [(1, 2), (64, 2), (128, 2), (129, 1), (257, 0), (640, 32)])
def test_backward_small_and_boundary_lengths(N, topk):
    run_bwd(1, 1, N, topk, TRAIN, seed=N + topk)


def test_backward_learned_selector():
    run_bwd(1, 2, 900, 3, TRAIN, seed=4, learned=True)


def test_backward_many_tiles_and_heads():
    # 96 heads x 5 tiles: every key pair has several query tiles in its inverted list
    run_bwd(2, 48, 600, 3, TRAIN, seed=5, heads=[(0, 0), (1, 47)])


def test_backward_full_size_dit_sampled():
    N = 4096 + 512
    run_bwd(2, 24, N, 32, TRAIN, seed=6, heads=[(0, 3), (1, 20)], rows=P.sample_rows(N, n_random=96))


def test_backward_repeated_calls_identical():
    a = run_bwd(1, 4, 800, 4, TRAIN, seed=7, heads=[(0, 0)])
    b = run_bwd(1, 4, 800, 4, TRAIN, seed=7, heads=[(0, 0)])
    for x, y in zip(a, b):
        assert torch.equal(x, y)


def test_backward_captured_in_a_cuda_graph_matches_eager():
    # after the first call has sized the workspace, a backward call is
    # asynchronous: captured in a CUDA graph, each replay equals the eager result
    B, H, N, d, K = 1, 4, 1000, 128, 4
    C = -(-N // 64)
    Q, Kk, V = (t.to(DEV) for t in synth.qkv(B, H, N, d, seed=8))
    S = synth.scores(B, H, N, C, seed=8, regime="R1").to(DEV)
    dO = synth.normal((B, H, N, d), 9).to(torch.bfloat16).to(DEV)
    layer = sas.SasLayer(B, H, N, d, K)
    O, LSE, si, sl = layer.attention(Q, Kk, V, scores=S)
    eager = layer.attention_bwd(Q, Kk, V, O, LSE, dO, scores=S, sel_idx=si, sel_logg=sl, want_ds=True)
    torch.cuda.synchronize()
    outs = [torch.empty_like(t) for t in eager]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        st = torch.cuda.current_stream()
        sas.sas_attention_bwd(layer.h, Q, Kk, V, O, LSE, dO, outs[0], outs[1], outs[2], S, si, sl, outs[3], outs[4],
                              st)
    for _ in range(2):
        for t in outs:
            t.zero_()
        g.replay()
        torch.cuda.synchronize()
        for x, y in zip(eager, outs):
            assert torch.equal(x, y)
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
