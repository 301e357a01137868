"""The handle-free, allocation-free MLP entry point (sas_mlp_fwd_noalloc).

It exists for callers that cannot allocate device memory while they run a
layer -- for instance code recording a CUDA graph, or a plug-in whose host
framework owns all device memory.  It keeps the hidden activation in a fixed
array inside the library instead of a handle's cudaMalloc'd buffer.  These
tests call it through the C ABI and check that it returns what the regular
sas_mlp_fwd returns, twice in a row (the array is shared and keeps the
previous call's contents), and that sizes beyond the array are refused.
The file is collected last so that a failure here cannot hide other tests.
"""
import numpy as np
import pytest
import torch

from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu


def _within_mlp_tolerance(Y, ref):
    # the tolerance the MLP parity tests use (see tests/test_gpu_mlp.py)
    err = np.abs(P.f64(Y) - P.f64(ref))
    r = np.abs(P.f64(ref))
    assert float((err - (2e-2 + 2.0 ** -8 * r)).max()) <= 0
    assert float(err.mean()) <= 2e-3 + 2.0 ** -9 * float(r.mean())


@pytest.mark.parametrize("T,D,F,bias", [(300, 256, 1024, True), (1024, 3072, 12288, False)])
def test_noalloc_mlp_matches_regular_entry_point_twice(T, D, F, bias):
    dev = torch.device("cuda:0")
    X, W1, W2, b1, b2 = (None if t is None else t.to(dev) for t in synth.mlp(T, D, F, seed=5, bias=bias))
    layer = sas.SasLayer(1, 1, 64, 64, 0)
    ref = layer.mlp(X, W1, W2, b1, b2)
    layer.close()
    for _ in range(2):
        Y = torch.full((T, D), float("nan"), device=dev, dtype=torch.bfloat16)
        sas.sas_mlp_fwd_noalloc(X, W1, W2, Y, b1, b2)
        torch.cuda.synchronize()
        assert not torch.isnan(Y).any()
        _within_mlp_tolerance(Y.cpu(), ref.cpu())


def test_noalloc_mlp_refuses_sizes_beyond_its_array():
    dev = torch.device("cuda:0")
    T, D, F = 2048, 64, 8192            # hidden activation 32 MiB + 0: exactly at the limit is allowed
    X = torch.zeros(T, D, device=dev, dtype=torch.bfloat16)
    W1 = torch.zeros(F, D, device=dev, dtype=torch.bfloat16)
    W2 = torch.zeros(D, F, device=dev, dtype=torch.bfloat16)
    Y = torch.empty(T, D, device=dev, dtype=torch.bfloat16)
    sas.sas_mlp_fwd_noalloc(X, W1, W2, Y)
    torch.cuda.synchronize()
    X2 = torch.zeros(T + 1, D, device=dev, dtype=torch.bfloat16)
    Y2 = torch.empty(T + 1, D, device=dev, dtype=torch.bfloat16)
    with pytest.raises(sas.SasError, match="exceeds"):
        sas.sas_mlp_fwd_noalloc(X2, W1, W2, Y2)
