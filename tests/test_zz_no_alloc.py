"""The handle-free, allocation-free MLP entry point (sas_mlp_fwd_noalloc).

It exists for callers that cannot allocate device memory while they run a
layer -- for instance code recording a CUDA graph, or a plug-in whose host
framework owns all device memory.  It keeps the hidden activation in a fixed
array inside the library instead of a handle's cudaMalloc'd buffer.  These
tests call it through the C ABI, twice in a row (the array is shared and
keeps the previous call's contents), and check each result against the
regular sas_mlp_fwd and, on sampled rows, against the fp64 oracle; after each
call the entry point's own status word (sas_mlp_noalloc_get_device_status)
must read SAS_OK.  Sizes beyond the array are refused.  The file is
collected last so that a failure here cannot hide other tests.
"""
import numpy as np
import pytest
import torch

from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu


def _within_mlp_tolerance(Y, ref):
    # the tolerance the MLP parity tests use (tests/test_gpu_mlp.py): bf16
    # output rounding of values up to about +-9 on top of 2e-2 / 2e-3
    err = np.abs(P.f64(Y) - ref)
    r = np.abs(ref)
    assert float((err - (2e-2 + 2.0 ** -8 * r)).max()) <= 0
    assert float(err.mean()) <= 2e-3 + 2.0 ** -9 * float(r.mean())


@pytest.mark.parametrize("T,D,F,bias", [(300, 256, 1024, True), (1024, 3072, 12288, False)])
def test_noalloc_mlp_matches_regular_entry_point_and_oracle_twice(T, D, F, bias):
    dev = torch.device("cuda:0")
    host = synth.mlp(T, D, F, seed=5, bias=bias)
    X, W1, W2, b1, b2 = (None if t is None else t.to(dev) for t in host)
    layer = sas.SasLayer(1, 1, 64, 64, 0)
    ref = layer.mlp(X, W1, W2, b1, b2)
    layer.close()
    rows = np.unique(np.concatenate([[0, T - 1], np.random.default_rng(0).integers(0, T, size=48)]))
    f = lambda t: None if t is None else P.f64(t)
    yref = OR.gelu_mlp(f(host[0]), f(host[1]), f(host[2]), f(host[3]), f(host[4]), rows=rows)
    assert sas.sas_mlp_noalloc_get_device_status() == sas.SAS_OK   # clears anything left before
    for _ in range(2):
        # Y is followed in memory by a NaN guard that the call must leave alone
        buf = torch.full((T * D + 4096,), float("nan"), device=dev, dtype=torch.bfloat16)
        Y = buf[:T * D].view(T, D)
        sas.sas_mlp_fwd_noalloc(X, W1, W2, Y, b1, b2)
        assert sas.sas_mlp_noalloc_get_device_status() == sas.SAS_OK
        assert not torch.isnan(Y).any()
        assert bool(torch.isnan(buf[T * D:]).all())
        _within_mlp_tolerance(Y.cpu(), P.f64(ref.cpu()))
        _within_mlp_tolerance(Y.cpu()[rows], yref)


def test_noalloc_mlp_refuses_sizes_beyond_its_array():
    dev = torch.device("cuda:0")
    T, D, F = 2048, 64, 8192            # hidden activation 32 MiB + 0: exactly at the limit is allowed
    X = torch.zeros(T, D, device=dev, dtype=torch.bfloat16)
    W1 = torch.zeros(F, D, device=dev, dtype=torch.bfloat16)
    W2 = torch.zeros(D, F, device=dev, dtype=torch.bfloat16)
    Y = torch.empty(T, D, device=dev, dtype=torch.bfloat16)
    sas.sas_mlp_fwd_noalloc(X, W1, W2, Y)
    assert sas.sas_mlp_noalloc_get_device_status() == sas.SAS_OK
    X2 = torch.zeros(T + 1, D, device=dev, dtype=torch.bfloat16)
    Y2 = torch.empty(T + 1, D, device=dev, dtype=torch.bfloat16)
    with pytest.raises(sas.SasError, match="exceeds"):
        sas.sas_mlp_fwd_noalloc(X2, W1, W2, Y2)


def test_noalloc_mlp_captured_in_a_cuda_graph():
    # the entry point's purpose: a CUDA graph capture fails on any allocation,
    # so a call captured (after one warm-up call outside the capture, which sets
    # the kernels' attributes) and replayed must reproduce the eager result
    dev = torch.device("cuda:0")
    T, D, F = 300, 256, 1024
    X, W1, W2, b1, b2 = (t.to(dev) for t in synth.mlp(T, D, F, seed=6, bias=True))
    Y = torch.empty(T, D, device=dev, dtype=torch.bfloat16)
    sas.sas_mlp_fwd_noalloc(X, W1, W2, Y, b1, b2)
    torch.cuda.synchronize()
    assert sas.sas_mlp_noalloc_get_device_status() == sas.SAS_OK
    eager = Y.clone()
    Y.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        sas.sas_mlp_fwd_noalloc(X, W1, W2, Y, b1, b2)
    for _ in range(2):
        Y.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(Y, eager)
    assert sas.sas_mlp_noalloc_get_device_status() == sas.SAS_OK
