"""Pins of the backward oracle: torch autograd through a dense masked form of
the same forward (with the gates computed from the scores by log_softmax and
the Top-K choice held fixed), central finite differences of the pinned forward
oracle, and the paper's closed form of the gate gradient (App. D).  CPU only."""
import math

import numpy as np
import pytest
import torch

from oracle import backward_oracle as BO
from oracle import sas_oracle as O


def _inputs(N, d, seed, C=None):
    rng = np.random.default_rng(seed)
    Q, K, V, dO = (rng.standard_normal((N, d)) for _ in range(4))
    C = C or -(-N // 8)
    s = rng.standard_normal((N, C))
    return Q, K, V, dO, s


def _torch_dense(Q, K, V, s, b, topk, sm_scale):
    """Dense masked attention whose bias on kept blocks is log_softmax(s) over
    the row's history; autograd gives dQ, dK, dV and ds."""
    N, d = Q.shape
    t = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    q, k, v, st = t(Q), t(K), t(V), t(s)
    rows = []
    for i in range(N):
        c = i // b
        bias = torch.full((N,), -math.inf, dtype=torch.float64)
        if c:
            lg = torch.log_softmax(st[i, :c], dim=0)
            sel = O.topk_blocks(s[i, :c], topk)
            bias = bias.clone()
            for m in sel:
                bias = torch.cat([bias[:m * b], lg[m].expand(b), bias[(m + 1) * b:]])
        bias = torch.cat([bias[:c * b], torch.zeros(i + 1 - c * b, dtype=torch.float64), bias[i + 1:]])
        rows.append(bias)
    Bm = torch.stack(rows)
    Z = sm_scale * q @ k.T + Bm
    P = torch.softmax(Z, dim=1)
    return q, k, v, st, P @ v


@pytest.mark.parametrize("N,topk,seed", [(37, 2, 0), (64, 1, 1), (50, 3, 2), (9, 0, 3)])
def test_backward_equals_torch_autograd_of_dense_form(N, topk, seed):
    b, d = 8, 6
    Q, K, V, dO, s = _inputs(N, d, seed)
    sm = 1 / math.sqrt(d)
    q, k, v, st, Ot = _torch_dense(Q, K, V, s, b, topk, sm)
    (Ot * torch.tensor(dO)).sum().backward()
    r = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk)
    assert np.allclose(r["dQ"], q.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dK"], k.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dV"], v.grad.numpy(), atol=1e-12)
    C = r["ds"].shape[1]
    gs = st.grad.numpy() if st.grad is not None else np.zeros_like(s)   # K = 0: the scores are unused
    assert np.allclose(r["ds"], gs[:, :C], atol=1e-12)
    assert np.all(gs[:, C:] == 0)


def test_backward_central_finite_differences():
    b, d, N, topk = 4, 3, 14, 1
    Q, K, V, dO, s = _inputs(N, d, 7, C=4)

    def loss(Qx, Kx, Vx, sx):
        return float((O.sas_attention_head(Qx, Kx, Vx, sx, b, topk)["O"] * dO).sum())

    r = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk)
    h = 1e-6
    for name, X, grad in [("Q", Q, r["dQ"]), ("K", K, r["dK"]), ("V", V, r["dV"]), ("s", s, None)]:
        G = np.zeros_like(X)
        for idx in np.ndindex(X.shape):
            Xp, Xm = X.copy(), X.copy()
            Xp[idx] += h
            Xm[idx] -= h
            args_p = [Q, K, V, s]
            args_m = [Q, K, V, s]
            pos = "QKVs".index(name)
            args_p[pos], args_m[pos] = Xp, Xm
            G[idx] = (loss(*args_p) - loss(*args_m)) / (2 * h)
        ref = grad if grad is not None else np.pad(r["ds"], ((0, 0), (0, s.shape[1] - r["ds"].shape[1])))
        # the Top-K choice must not flip inside the difference step (scores well separated here)
        assert np.allclose(G, ref, atol=1e-6), name


def test_gate_gradient_closed_form_of_the_paper():
    # App. D: dg_m = sum_{i in B_m} (p_i / g_m) dO.(v_i - o); dlogg_m = g_m dg_m
    b, d, N, topk = 8, 5, 40, 2
    Q, K, V, dO, s = _inputs(N, d, 11)
    r = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk)
    fwd = O.sas_attention_head(Q, K, V, s, b, topk)
    for i in range(N):
        keys, bias, _, sel, lg = O._row_keys_and_bias(i, s[i], b, topk, O.MODE_TRAIN_SOFT)
        z = (K[keys] @ Q[i]) / math.sqrt(d) + bias
        p = np.exp(z - z.max())
        p /= p.sum()
        for e, m in enumerate(sel):
            g = math.exp(lg[e])
            blk = slice(e * b, (e + 1) * b)
            dg = ((p[blk] / g) * (V[keys][blk] @ dO[i] - fwd["O"][i] @ dO[i])).sum()
            assert math.isclose(r["dlogg"][i, e], g * dg, rel_tol=1e-10, abs_tol=1e-12)


def test_score_gradient_sums_to_zero_and_inference_has_none():
    # softmax gates: a common shift of a row's scores changes nothing, so the
    # score gradient of every row sums to zero; inference mode has no gates
    b, d, N, topk = 8, 4, 45, 2
    Q, K, V, dO, s = _inputs(N, d, 5)
    r = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk)
    assert np.allclose(r["ds"].sum(axis=1), 0, atol=1e-12)
    ri = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk, mode=O.MODE_INFER_HARD)
    assert np.all(ri["ds"] == 0) and np.all(ri["dlogg"] == 0)


def test_delta_is_rowsum_of_o_times_do():
    b, d, N, topk = 8, 4, 30, 2
    Q, K, V, dO, s = _inputs(N, d, 9)
    r = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk)
    fwd = O.sas_attention_head(Q, K, V, s, b, topk)
    assert np.allclose(r["Delta"], (fwd["O"] * dO).sum(axis=1), atol=1e-13)


def test_gqa_backward_equals_autograd_with_shared_keys_values_and_gates():
    # one group of G = 2 heads over shared K, V and scores: torch autograd through the
    # dense masked form of both heads (the same shared tensors feed both) gives the
    # sums the GQA oracle must produce
    b, d, N, topk, G = 8, 4, 30, 2, 2
    rng = np.random.default_rng(21)
    Q = rng.standard_normal((G, N, d))
    K, V = rng.standard_normal((1, N, d)), rng.standard_normal((1, N, d))
    s = rng.standard_normal((1, N, -(-N // b)))
    dO = rng.standard_normal((G, N, d))
    sm = 1 / math.sqrt(d)
    t = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    kk, vv, st = t(K[0]), t(V[0]), t(s[0])
    qs = [t(Q[h]) for h in range(G)]
    loss = 0
    for h in range(G):
        rows = []
        for i in range(N):
            c = i // b
            bias = torch.full((N,), -math.inf, dtype=torch.float64)
            if c:
                lg = torch.log_softmax(st[i, :c], dim=0)
                for m in O.topk_blocks(s[0, i, :c], topk):
                    bias = torch.cat([bias[:m * b], lg[m].expand(b), bias[(m + 1) * b:]])
            bias = torch.cat([bias[:c * b], torch.zeros(i + 1 - c * b, dtype=torch.float64), bias[i + 1:]])
            rows.append(bias)
        P = torch.softmax(sm * qs[h] @ kk.T + torch.stack(rows), dim=1)
        loss = loss + ((P @ vv) * torch.tensor(dO[h])).sum()
    loss.backward()
    r = BO.sas_attention_bwd_gqa(Q, K, V, s, dO, b, topk)
    for h in range(G):
        assert np.allclose(r["dQ"][h], qs[h].grad.numpy(), atol=1e-12)
    assert np.allclose(r["dK"][0], kk.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dV"][0], vv.grad.numpy(), atol=1e-12)
    assert np.allclose(r["ds"][0], st.grad.numpy()[:, :r["ds"].shape[2]], atol=1e-12)


def test_gqa_backward_with_one_head_per_group_is_the_head_backward():
    b, d, N, topk = 8, 3, 26, 2
    rng = np.random.default_rng(22)
    Q, K, V, dO = (rng.standard_normal((2, N, d)) for _ in range(4))
    s = rng.standard_normal((2, N, 4))
    r = BO.sas_attention_bwd_gqa(Q, K, V, s, dO, b, topk)
    for h in range(2):
        m = BO.sas_attention_bwd_head(Q[h], K[h], V[h], s[h], dO[h], b, topk)
        for f in ("dQ", "dK", "dV", "dlogg", "ds"):
            assert np.allclose(r[f][h], m[f], atol=1e-13), f


def test_packed_backward_equals_autograd_of_the_packed_forward_oracle():
    # central finite differences of the packed forward oracle (through K of both
    # sequences and the scores) against the packed backward: the sequences' block
    # partitions start at their own first rows, and no gradient crosses them
    b, d, topk = 4, 3, 1
    rng = np.random.default_rng(23)
    lens = [9, 11]
    T = sum(lens)
    cu = [0, 9, 20]
    Q, K, V, dO = (rng.standard_normal((1, T, d)) for _ in range(4))
    s = rng.standard_normal((1, T, 3))
    r = BO.sas_attention_bwd_varlen(Q, K, V, s, dO, cu, b, topk)

    def loss(Kx, sx):
        return float((O.sas_attention_varlen(Q, Kx, V, cu, b, topk, sx)["O"] * dO).sum())

    h = 1e-6
    for name, X, ref in (("K", K, r["dK"]), ("s", s, r["ds"])):
        G = np.zeros_like(X)
        for idx in np.ndindex(X.shape):
            Xp, Xm = X.copy(), X.copy()
            Xp[idx] += h
            Xm[idx] -= h
            args_p = (Xp, s) if name == "K" else (K, Xp)
            args_m = (Xm, s) if name == "K" else (K, Xm)
            G[idx] = (loss(*args_p) - loss(*args_m)) / (2 * h)
        assert np.allclose(G, ref, atol=1e-6), name
