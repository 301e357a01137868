"""GPU parity of the dense GELU MLP sublayer against the fp64 oracle, through
the C ABI.

Tolerance: the output is bf16, and with the benchmark's initialisation its
values reach about +-9, where one bf16 step is 2^-4; no bf16 result can be
closer to the exact value than half a step.  The bound is therefore
|err| <= 2e-2 + 2^-8 |ref| per element (2^-8 |ref| is half a bf16 step at
the value's magnitude, the rest allows fp32 accumulation and the rare hidden
activation that the two sides round to neighbouring bf16 values), and a mean
error of at most 2e-3 + 2^-9 mean|ref| (the average bf16 output rounding).
"""
import numpy as np
import pytest
import torch

from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu


def _check(Y, ref):
    err = np.abs(Y - ref)
    bound = 2e-2 + 2.0 ** -8 * np.abs(ref)
    worst = float((err - bound).max())
    assert worst <= 0, f"max excess over bound {worst:.3e}; max abs err {err.max():.3e}"
    mean_bound = 2e-3 + 2.0 ** -9 * float(np.abs(ref).mean())
    assert float(err.mean()) <= mean_bound, f"mean abs err {err.mean():.3e} > {mean_bound:.3e}"


def _run(T, D, F, bias, rows=None, seed=0):
    X, W1, W2, b1, b2 = synth.mlp(T, D, F, seed=seed, bias=bias)
    layer = sas.SasLayer(1, 1, 64, 64, 0)
    cu = lambda t: None if t is None else t.cuda()
    Y = layer.mlp(cu(X), cu(W1), cu(W2), cu(b1), cu(b2)).cpu()
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    f = lambda t: None if t is None else P.f64(t)
    ref = OR.gelu_mlp(f(X), f(W1), f(W2), f(b1), f(b2), rows=rows)
    Yg = P.f64(Y) if rows is None else P.f64(Y)[rows]
    _check(Yg, ref)


def test_mlp_tiny_block():
    _run(256, 256, 1024, bias=False)


def test_mlp_ragged_tokens_with_bias():
    _run(300, 192, 320, bias=True, seed=1)


def test_mlp_single_token():
    _run(1, 128, 256, bias=True, seed=2)


def test_mlp_stress_config_sampled_rows():
    # MLP stress shape: 16384 tokens, 3072 -> 12288 -> 3072
    rows = np.random.default_rng(0).choice(16384, size=48, replace=False)
    rows = np.concatenate([rows, [0, 127, 128, 16383]])
    _run(16384, 3072, 12288, bias=False, rows=rows)


def test_mlp_multi_tile_ragged_rows_with_bias():
    # eight 128-row tiles, the last with 104 rows; N = 2048 and 512 give several
    # 256-wide output tiles per row block
    _run(1000, 512, 2048, bias=True, seed=3)
