"""Failure paths of the real kernels, without a GPU fault.

Every wait inside the library's kernels is bounded.  With the handle's
main-loop budget cut to one SM cycle (sas_set_wait_limit), the selection,
attention and GEMM kernels give up at their first wait that is not already
satisfied: they record SAS_ERR_TIMEOUT in the device status word, drain their
own in-flight copies and tensor-core work (under the normal budget), free
their tensor memory and return.  The test checks the status, that the context
still runs work, and that the same handle gives the correct result again once
the default budget is restored."""
import numpy as np
import pytest
import torch

from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _layer_inputs():
    B, H, N, d, K = 1, 8, 4608, 128, 32
    Q, Kk, V = synth.qkv(B, H, N, d, seed=3, regime="R2")
    Wq, Wk = synth.selector_weights(H, d, d, seed=3)
    X, W1, W2, _, _ = synth.mlp(2048, 512, 2048, seed=3)
    return (B, H, N, d, K), [t.to(DEV) for t in (Q, Kk, V, Wq, Wk, X, W1, W2)], (Q, Kk, V, Wq, Wk)


def test_kernels_give_up_report_timeout_and_recover():
    (B, H, N, d, K), (Q, Kk, V, Wq, Wk, X, W1, W2), host = _layer_inputs()
    layer = sas.SasLayer(B, H, N, d, K, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d)
    ref = layer.attention(Q, Kk, V, Wq=Wq, Wk=Wk)
    yref = layer.mlp(X, W1, W2)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == sas.SAS_OK

    # attention (block summaries, selection, attention kernels) under a 1-cycle budget
    sas.sas_set_wait_limit(layer.h, 1)
    layer.attention(Q, Kk, V, Wq=Wq, Wk=Wk)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == sas.SAS_ERR_TIMEOUT
    # the MLP's two GEMM kernels under the same budget
    layer.mlp(X, W1, W2)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == sas.SAS_ERR_TIMEOUT

    # the context still runs work
    x = torch.arange(1 << 20, device=DEV, dtype=torch.float32)
    assert float(x.sum()) == float((1 << 20) * ((1 << 20) - 1) // 2)

    # the same handle computes the right result again with the default budget
    sas.sas_set_wait_limit(layer.h, 0)
    out = layer.attention(Q, Kk, V, Wq=Wq, Wk=Wk)
    y = layer.mlp(X, W1, W2)
    torch.cuda.synchronize()
    assert sas.sas_get_device_status(layer.h) == sas.SAS_OK
    layer.close()
    for a, b in zip(out, ref):
        assert torch.equal(a, b)            # the kernels are deterministic
    assert torch.equal(y, yref)
    Qh, Kh, Vh, Wqh, Wkh = host
    rows = P.sample_rows(N, n_random=64)
    s = P.oracle_scores(Qh, Kh, Wqh, Wkh, 0, 5)
    r = OR.sas_attention_head(P.f64(Qh[0, 5]), P.f64(Kh[0, 5]), P.f64(Vh[0, 5]), s, 64, K, rows=rows)
    tol = P.selector_score_bound(Qh, Kh, Wqh, Wkh, 0, 5, d, rows=rows)
    _, _, mism = P.check_selection_rows(out[2][0, 5].cpu().numpy()[rows][:, :K], s[rows], rows, K, tol)
    keep = ~mism
    P.compare_o(P.f64(out[0][0, 5].cpu())[rows][keep], r["O"][keep], "O[0,5]")


def test_wait_limit_rejects_negative_budgets():
    layer = sas.SasLayer(1, 1, 128, 64, 2)
    with pytest.raises(sas.SasError):
        sas.sas_set_wait_limit(layer.h, -5)
    layer.close()
