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


def _torch_dense(Q, K, V, s, b, topk, sm_scale, act=O.GATE_SOFTMAX):
    """Dense masked attention whose bias on kept blocks is log g of the gate
    activation (softmax: log_softmax(s) over the row's history; sigmoid:
    logsigmoid(s); raw logit: s); autograd gives dQ, dK, dV and ds."""
    N, d = Q.shape
    t = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    q, k, v, st = t(Q), t(K), t(V), t(s)
    rows = []
    for i in range(N):
        c = i // b
        bias = torch.full((N,), -math.inf, dtype=torch.float64)
        if c:
            if act == O.GATE_SIGMOID:
                lg = torch.nn.functional.logsigmoid(st[i, :c])
            elif act == O.GATE_LOGIT:
                lg = st[i, :c]
            else:
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


# ---------------------------------------------------------------- full scope

@pytest.mark.parametrize("N,seed", [(41, 31), (64, 32)])
def test_full_scope_backward_equals_autograd_with_every_block_gated(N, seed):
    # Sec. 4.2 full scope: no Top-K, every historical block enters with log g =
    # log_softmax(s); the dense masked form keeping all blocks gives its gradients
    b, d = 8, 5
    Q, K, V, dO, s = _inputs(N, d, seed)
    sm = 1 / math.sqrt(d)
    C = -(-N // b)
    q, k, v, st, Ot = _torch_dense(Q, K, V, s, b, C, sm)
    (Ot * torch.tensor(dO)).sum().backward()
    r = BO.sas_attention_bwd_full_head(Q, K, V, s, dO, b)
    assert np.allclose(r["dQ"], q.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dK"], k.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dV"], v.grad.numpy(), atol=1e-12)
    assert np.allclose(r["ds"], st.grad.numpy()[:, :C], atol=1e-12)
    # dlogg is indexed by block (every block is kept): the paper's closed form
    # dlogg_m = g_m dg_m, dg_m = sum_{j in B_m} (p_j / g_m) dO.(v_j - o) (App. D)
    assert r["dlogg"].shape == (N, C)
    fwd = O.sas_attention_full_scope(Q, K, V, s, b)
    for i in range(b, N):
        c = i // b
        lg = O.log_gates(s[i, :c])
        keys = np.arange(i + 1)
        z = sm * (K[keys] @ Q[i]) + np.concatenate([np.repeat(lg, b), np.zeros(i + 1 - c * b)])
        p = np.exp(z - z.max())
        p /= p.sum()
        for m in range(c):
            blk = slice(m * b, (m + 1) * b)
            g = math.exp(lg[m])
            dg = ((p[blk] / g) * (V[blk] @ dO[i] - fwd["O"][i] @ dO[i])).sum()
            assert math.isclose(r["dlogg"][i, m], g * dg, rel_tol=1e-9, abs_tol=1e-12)


# -------------------------------------------------------- hard gate with STE

def _torch_ste(Q, K, V, s, b, topk, sm_scale):
    """Dense form of the hard Top-K gate under the straight-through estimator:
    row i weighs token j of historical block m by g^hat_m exp(z_j), the current
    block by exp(z_j), with g^hat = stopgrad(g^hard - g) + g, g = softmax(s_i)
    over the row's history.  Returns the leaves, O and each row's g^hat (its
    gradient retained)."""
    N, d = Q.shape
    t = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    q, k, v, st = t(Q), t(K), t(V), t(s)
    Z = sm_scale * q @ k.T
    outs, ghats = [], []
    for i in range(N):
        c = i // b
        w_hist = []
        if c:
            g = torch.softmax(st[i, :c], dim=0)
            hard = torch.zeros(c, dtype=torch.float64)
            hard[O.topk_blocks(s[i, :c], topk)] = 1.0
            gh = (hard - g).detach() + g
            gh.retain_grad()
            ghats.append(gh)
            w_hist = [gh.repeat_interleave(b)]
        else:
            ghats.append(None)
        zi = Z[i, :i + 1]
        w = torch.exp(zi - zi.max().detach())
        wt = torch.cat(w_hist + [torch.ones(i + 1 - c * b, dtype=torch.float64)]) * w
        outs.append((wt @ v[:i + 1]) / wt.sum())
    return q, k, v, st, torch.stack(outs), ghats


@pytest.mark.parametrize("N,topk,seed", [(37, 2, 41), (50, 1, 42), (33, 0, 43)])
def test_ste_backward_equals_autograd_through_the_estimator(N, topk, seed):
    b, d = 8, 5
    Q, K, V, dO, s = _inputs(N, d, seed)
    sm = 1 / math.sqrt(d)
    q, k, v, st, Ot, ghats = _torch_ste(Q, K, V, s, b, topk, sm)
    (Ot * torch.tensor(dO)).sum().backward()
    r = BO.sas_attention_bwd_ste_head(Q, K, V, s, dO, b, topk)
    # the forward is the hard one
    assert np.allclose(Ot.detach().numpy(), O.sas_attention_head(Q, K, V, s, b, topk, O.MODE_INFER_HARD)["O"],
                       atol=1e-12)
    assert np.allclose(r["dQ"], q.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dK"], k.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dV"], v.grad.numpy(), atol=1e-12)
    C = r["ds"].shape[1]
    assert np.allclose(r["ds"], st.grad.numpy()[:, :C], atol=1e-12)
    for i, gh in enumerate(ghats):
        if gh is not None:
            assert np.allclose(r["dg"][i, :gh.shape[0]], gh.grad.numpy(), atol=1e-12)
    # x = g dg, and ds = x - g sum(x) (the sparse score-gradient formula applied to x)
    for i in range(N):
        c = i // b
        if c:
            g = np.exp(O.log_gates(s[i, :c]))
            assert np.allclose(r["x"][i, :c], g * r["dg"][i, :c], atol=1e-14)
            assert np.allclose(r["ds"][i, :c], r["x"][i, :c] - g * r["x"][i, :c].sum(), atol=1e-12)


def test_ste_gate_weight_of_a_dropped_block_is_unbounded():
    # Eq. rank_unbounded: a dropped block whose logits outscore the attended set
    # gets p~ = exp(z - LSE_S) > 1, so its dg grows with exp(z - max_S z)
    b, d, N, topk = 4, 2, 12, 1
    Q = np.zeros((N, d)); Q[:, 0] = 1.0
    K = np.zeros((N, d)); K[0:4, 0] = 6.0          # block 0: large logits for every query
    V = np.zeros((N, d)); V[0:4, 1] = 1.0
    dO = np.zeros((N, d)); dO[:, 1] = 1.0
    s = np.zeros((N, 3)); s[:, 1] = 5.0            # the selector keeps block 1, drops block 0
    r = BO.sas_attention_bwd_ste_head(Q, K, V, s, dO, b, topk, sm_scale=1.0)
    i = N - 1                                      # row 11: blocks 0, 1 historical, block 1 kept
    assert O.topk_blocks(s[i, :2], topk).tolist() == [1]
    # the attended set holds block 1 (z = 0) and row i's own block (z = 0): LSE_S = log 8
    pt = math.exp(6.0 - math.log(8.0))
    assert pt > 1
    assert math.isclose(r["dg"][i, 0], 4 * pt * (1.0 - 0.0), rel_tol=1e-12)


def test_ste_gqa_is_the_sum_over_heads():
    b, d, N, topk = 8, 3, 30, 2
    rng = np.random.default_rng(44)
    Q, dO = rng.standard_normal((4, N, d)), rng.standard_normal((4, N, d))
    K, V = rng.standard_normal((2, N, d)), rng.standard_normal((2, N, d))
    s = rng.standard_normal((2, N, 4))
    r = BO.sas_attention_bwd_ste_gqa(Q, K, V, s, dO, b, topk)
    for g in range(2):
        parts = [BO.sas_attention_bwd_ste_head(Q[h], K[g], V[g], s[g], dO[h], b, topk) for h in (2 * g, 2 * g + 1)]
        assert np.allclose(r["dK"][g], parts[0]["dK"] + parts[1]["dK"], atol=1e-13)
        assert np.allclose(r["dg"][g], parts[0]["dg"] + parts[1]["dg"], atol=1e-13)
        for i in range(N):
            c = i // b
            if c:
                gt = np.exp(O.log_gates(s[g, i, :c]))
                dgi = r["dg"][g, i, :c]
                assert np.allclose(r["ds"][g, i, :c], gt * (dgi - (gt * dgi).sum()), atol=1e-13)


# ------------------------------------------- other gate activations (inner)

@pytest.mark.parametrize("act", [O.GATE_SIGMOID, O.GATE_LOGIT])
@pytest.mark.parametrize("N,topk,seed", [(37, 2, 51), (50, 3, 52)])
def test_other_activations_backward_equals_autograd(act, N, topk, seed):
    # Sec. 4.2 gate activation: independent gates, so only kept blocks get a
    # score gradient, through d log g / ds (sigmoid: 1 - g; raw logit: 1)
    b, d = 8, 5
    Q, K, V, dO, s = _inputs(N, d, seed)
    sm = 1 / math.sqrt(d)
    q, k, v, st, Ot = _torch_dense(Q, K, V, s, b, topk, sm, act)
    assert np.allclose(Ot.detach().numpy(), O.sas_attention_head(Q, K, V, s, b, topk, act=act)["O"], atol=1e-12)
    (Ot * torch.tensor(dO)).sum().backward()
    r = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk, act=act)
    assert np.allclose(r["dQ"], q.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dK"], k.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dV"], v.grad.numpy(), atol=1e-12)
    C = r["ds"].shape[1]
    assert np.allclose(r["ds"], st.grad.numpy()[:, :C], atol=1e-12)
    # dropped blocks get none, unlike the softmax gates
    for i in range(N):
        c = i // b
        dropped = np.setdiff1d(np.arange(c), O.topk_blocks(s[i, :c], topk))
        assert np.all(r["ds"][i, dropped] == 0)


# ------------------------------------------------------- outer gate position

@pytest.mark.parametrize("act", [O.GATE_SOFTMAX, O.GATE_SIGMOID])
@pytest.mark.parametrize("N,topk,seed", [(37, 2, 61), (45, 3, 62)])
def test_outer_position_backward_equals_autograd(act, N, topk, seed):
    # Sec. 4.2 gate position: o = softmax(z) (g . V), z unbiased, each kept
    # block's value rows scaled by its gate (the current block by 1)
    b, d = 8, 5
    Q, K, V, dO, s = _inputs(N, d, seed)
    sm = 1 / math.sqrt(d)
    t = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    q, k, v, st = t(Q), t(K), t(V), t(s)
    outs = []
    for i in range(N):
        c = i // b
        mask = torch.full((N,), -math.inf, dtype=torch.float64)
        wts = torch.zeros(N, dtype=torch.float64)
        if c:
            lg = torch.nn.functional.logsigmoid(st[i, :c]) if act == O.GATE_SIGMOID else torch.log_softmax(st[i, :c], 0)
            for m in O.topk_blocks(s[i, :c], topk):
                mask = torch.cat([mask[:m * b], torch.zeros(b, dtype=torch.float64), mask[(m + 1) * b:]])
                wts = torch.cat([wts[:m * b], torch.exp(lg[m]).expand(b), wts[(m + 1) * b:]])
        mask = torch.cat([mask[:c * b], torch.zeros(i + 1 - c * b, dtype=torch.float64), mask[i + 1:]])
        wts = torch.cat([wts[:c * b], torch.ones(i + 1 - c * b, dtype=torch.float64), wts[i + 1:]])
        p = torch.softmax(sm * k @ q[i] + mask, dim=0)
        outs.append((p * wts) @ v)
    Ot = torch.stack(outs)
    fwd = O.sas_attention_head(Q, K, V, s, b, topk, act=act, pos=O.GATE_OUTER)
    assert np.allclose(Ot.detach().numpy(), fwd["O"], atol=1e-12)
    (Ot * torch.tensor(dO)).sum().backward()
    r = BO.sas_attention_bwd_head(Q, K, V, s, dO, b, topk, act=act, pos=O.GATE_OUTER)
    assert np.allclose(r["dQ"], q.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dK"], k.grad.numpy(), atol=1e-12)
    assert np.allclose(r["dV"], v.grad.numpy(), atol=1e-12)
    C = r["ds"].shape[1]
    assert np.allclose(r["ds"], st.grad.numpy()[:, :C], atol=1e-12)
    assert np.allclose(r["Delta"], (fwd["O"] * dO).sum(axis=1), atol=1e-13)
