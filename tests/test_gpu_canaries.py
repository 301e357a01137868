"""Output canaries (the stand-in for a memory checker): every output buffer of
every entry point is allocated with a guard region right behind it, filled
with a sentinel; after the call the guard must be untouched, so no kernel
writes past the end of the shapes the header documents."""
import numpy as np
import pytest
import torch

from paper_2609_13141_gb300 import sas, synth

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
GUARD = 4096   # elements behind each output


def guarded(shape, dtype):
    """(view, guard): a tensor of `shape` followed in memory by GUARD sentinel elements."""
    n = int(np.prod(shape))
    buf = torch.empty(n + GUARD, device=DEV, dtype=dtype)
    if dtype == torch.int32:
        buf.fill_(0x7EADBEEF)
    else:
        buf.fill_(float("nan"))
    return buf[:n].view(*shape), buf[n:]


def intact(guard):
    g = guard.view(torch.int16 if guard.dtype == torch.bfloat16 else torch.int32)
    ref = guarded((1,), guard.dtype)[1].view(g.dtype)[:g.numel()]
    return bool(torch.equal(g, ref))


def _check(*guards):
    torch.cuda.synchronize()
    for k, g in enumerate(guards):
        assert intact(g), f"output {k} was written past its end"


@pytest.mark.parametrize("selector,N,d", [(sas.SAS_SEL_SCORES_GIVEN, 1000, 128), (sas.SAS_SEL_MEANPOOL_PROJ, 777, 64)])
def test_attention_outputs_end_where_the_header_says(selector, N, d):
    B, H, K = 2, 3, 4
    Q, Kk, V = (t.to(DEV) for t in synth.qkv(B, H, N, d, seed=1, regime="R2"))
    kw = {}
    if selector == sas.SAS_SEL_SCORES_GIVEN:
        kw["scores"] = synth.scores(B, H, N, -(-N // 64), seed=1).to(DEV)
    else:
        kw["Wq"], kw["Wk"] = (t.to(DEV) for t in synth.selector_weights(H, d, d, seed=1))
    layer = sas.SasLayer(B, H, N, d, K, selector=selector, d_sel=d)
    O, gO = guarded((B, H, N, d), torch.bfloat16)
    L, gL = guarded((B, H, N), torch.float32)
    si, gi = guarded((B, H, N, K), torch.int32)
    sl, gl = guarded((B, H, N, K), torch.float32)
    sas.sas_attention_fwd(layer.h, Q, Kk, V, O, LSE=L, sel_idx=si, sel_logg=sl, **kw)
    _check(gO, gL, gi, gl)
    # the backward's outputs, after the forward of the same inputs (given scores, d = 128)
    if selector == sas.SAS_SEL_SCORES_GIVEN:
        dO = synth.normal((B, H, N, d), 5).to(torch.bfloat16).to(DEV)
        dQ, gq = guarded((B, H, N, d), torch.bfloat16)
        dK, gk = guarded((B, H, N, d), torch.bfloat16)
        dV, gv = guarded((B, H, N, d), torch.bfloat16)
        dl, gdl = guarded((B, H, N, K), torch.float32)
        ds, gds = guarded((B, H, N, -(-N // 64)), torch.float32)
        sas.sas_attention_bwd(layer.h, Q, Kk, V, O, L, dO, dQ, dK, dV, kw["scores"], si, sl, dl, ds)
        _check(gq, gk, gv, gdl, gds)
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()


def test_gqa_and_full_scope_outputs():
    B, H, Hkv, N, d, K = 1, 4, 2, 900, 128, 3
    Q = synth.qkv(B, H, N, d, seed=2)[0].to(DEV)
    _, Kk, V = (t.to(DEV) for t in synth.qkv(B, Hkv, N, d, seed=102))
    S = synth.scores(B, Hkv, N, -(-N // 64), seed=2).to(DEV)
    layer = sas.SasLayer(B, H, N, d, K, Hkv=Hkv)
    O, gO = guarded((B, H, N, d), torch.bfloat16)
    L, gL = guarded((B, H, N), torch.float32)
    si, gi = guarded((B, Hkv, N, K), torch.int32)
    sl, gl = guarded((B, Hkv, N, K), torch.float32)
    sas.sas_attention_fwd(layer.h, Q, Kk, V, O, S, LSE=L, sel_idx=si, sel_logg=sl)
    _check(gO, gL, gi, gl)
    # the GQA backward: dQ per query head, the rest per KV group
    dO = synth.normal((B, H, N, d), 6).to(torch.bfloat16).to(DEV)
    dQ, gq = guarded((B, H, N, d), torch.bfloat16)
    dK, gk = guarded((B, Hkv, N, d), torch.bfloat16)
    dV, gv = guarded((B, Hkv, N, d), torch.bfloat16)
    dl, gdl = guarded((B, Hkv, N, K), torch.float32)
    ds, gds = guarded((B, Hkv, N, -(-N // 64)), torch.float32)
    sas.sas_attention_bwd(layer.h, Q, Kk, V, O, L, dO, dQ, dK, dV, S, si, sl, dl, ds)
    _check(gq, gk, gv, gdl, gds)
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    full = sas.SasLayer(B, H, N, d, K, Hkv=Hkv, scope=sas.SAS_SCOPE_FULL)
    O, gO = guarded((B, H, N, d), torch.bfloat16)
    L, gL = guarded((B, H, N), torch.float32)
    sas.sas_attention_fwd(full.h, Q, Kk, V, O, S, LSE=L)
    _check(gO, gL)
    # the full scope's backward: a gate gradient for every block, [B, Hkv, N, C]
    C = -(-N // 64)
    dQ, gq = guarded((B, H, N, d), torch.bfloat16)
    dK, gk = guarded((B, Hkv, N, d), torch.bfloat16)
    dV, gv = guarded((B, Hkv, N, d), torch.bfloat16)
    dl, gdl = guarded((B, Hkv, N, C), torch.float32)
    ds, gds = guarded((B, Hkv, N, C), torch.float32)
    sas.sas_attention_bwd(full.h, Q, Kk, V, O, L, dO, dQ, dK, dV, S, None, None, dl, ds)
    _check(gq, gk, gv, gdl, gds)
    assert sas.sas_get_device_status(full.h) == 0
    full.close()
    # the hard gate under the straight-through estimator: hard forward, dense gate gradient
    ste = sas.SasLayer(B, H, N, d, K, Hkv=Hkv, mode=sas.SAS_MODE_TRAIN_HARD_STE)
    O, gO = guarded((B, H, N, d), torch.bfloat16)
    L, gL = guarded((B, H, N), torch.float32)
    si, gi = guarded((B, Hkv, N, K), torch.int32)
    sl, gl = guarded((B, Hkv, N, K), torch.float32)
    sas.sas_attention_fwd(ste.h, Q, Kk, V, O, S, LSE=L, sel_idx=si, sel_logg=sl)
    _check(gO, gL, gi, gl)
    dQ, gq = guarded((B, H, N, d), torch.bfloat16)
    dK, gk = guarded((B, Hkv, N, d), torch.bfloat16)
    dV, gv = guarded((B, Hkv, N, d), torch.bfloat16)
    dl, gdl = guarded((B, Hkv, N, C), torch.float32)
    ds, gds = guarded((B, Hkv, N, C), torch.float32)
    sas.sas_attention_bwd(ste.h, Q, Kk, V, O, L, dO, dQ, dK, dV, S, si, sl, dl, ds)
    _check(gq, gk, gv, gdl, gds)
    assert sas.sas_get_device_status(ste.h) == 0
    ste.close()


def test_varlen_outputs():
    lens, cap, H, Hkv, d, K = [300, 129, 64], 600, 2, 2, 128, 3
    Q = synth.qkv(1, H, cap, d, seed=3)[0][0].to(DEV)
    _, Kk, V = synth.qkv(1, Hkv, cap, d, seed=103)
    Kk, V = Kk[0].to(DEV), V[0].to(DEV)
    S = synth.scores(1, Hkv, cap, -(-max(lens) // 64), seed=3)[0].to(DEV)
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=DEV)
    layer = sas.SasLayer(1, H, cap, d, K, Hkv=Hkv, max_seqs=3, max_seqlen=max(lens))
    O, gO = guarded((H, cap, d), torch.bfloat16)
    L, gL = guarded((H, cap), torch.float32)
    si, gi = guarded((Hkv, cap, K), torch.int32)
    sl, gl = guarded((Hkv, cap, K), torch.float32)
    sas.sas_attention_fwd_varlen(layer.h, cu, Q, Kk, V, S, O, L, si, sl)
    _check(gO, gL, gi, gl)
    # the packed backward
    dO = synth.normal((H, cap, d), 7).to(torch.bfloat16).to(DEV)
    dQ, gq = guarded((H, cap, d), torch.bfloat16)
    dK, gk = guarded((Hkv, cap, d), torch.bfloat16)
    dV, gv = guarded((Hkv, cap, d), torch.bfloat16)
    dl, gdl = guarded((Hkv, cap, K), torch.float32)
    ds, gds = guarded((Hkv, cap, S.shape[-1]), torch.float32)
    sas.sas_attention_bwd(layer.h, Q, Kk, V, O, L, dO, dQ, dK, dV, S, si, sl, dl, ds)
    _check(gq, gk, gv, gdl, gds)
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()


def test_mlp_output():
    T, D, F = 333, 256, 1024
    X, W1, W2, b1, b2 = (t.to(DEV) for t in synth.mlp(T, D, F, seed=4, bias=True))
    layer = sas.SasLayer(1, 1, 64, 64, 0)
    Y, gY = guarded((T, D), torch.bfloat16)
    sas.sas_mlp_fwd(layer.h, X, W1, W2, Y, b1, b2)
    _check(gY)
    layer.close()


def test_decode_outputs():
    B, Hq, Hkv, d, K = 2, 8, 2, 128, 4
    lens = [700, 130]
    max_blocks = max(-(-n // 64) for n in lens) + 1
    table, npages = synth.decode_layout(lens, max_blocks, 5)
    Kc, Vc = synth.decode_cache(npages, Hkv, d, 5, device=DEV)
    q, kn, vn = synth.decode_queries(B, Hq, Hkv, d, 5, device=DEV)
    Wq, Wk = synth.decode_selector_weights(Hkv, Hq // Hkv, d, d, 5, device=DEV)
    Ksum = torch.zeros(B, Hkv, max_blocks, d, device=DEV, dtype=torch.bfloat16)
    dec = sas.SasDecoder(B, Hq, Hkv, d, K, max_blocks, npages, d_sel=d)
    tab = table.to(DEV)
    lens_t = torch.tensor(lens, dtype=torch.int32, device=DEV)
    dec.summarize(Kc, tab, lens_t - 1, Wk, Ksum)
    O, gO = guarded((B, Hq, d), torch.bfloat16)
    L, gL = guarded((B, Hq), torch.float32)
    si, gi = guarded((B, Hkv, K), torch.int32)
    dec.step(q, Kc, Vc, tab, lens_t, kn, vn, Wq, Wk, Ksum, out=(O, L, si))
    _check(gO, gL, gi)
    assert sas.sas_decode_get_device_status(dec.h) == 0
    dec.close()
