"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every function include/sas.h declares, and rejects bad configurations before
touching a device."""
import ctypes
import math
import subprocess

import pytest
import torch

from paper_2609_13141_gb300 import _build, sas


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return sas.lib()


def test_library_exports_every_declared_function(lib):
    names = sas.header_functions()
    assert "sas_attention_fwd" in names and "sas_mlp_fwd" in names and "sas_create" in names
    out = subprocess.run(["nm", "-D", "--defined-only", _build.LIB_PATH], capture_output=True, text=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if line.strip()}
    missing = [n for n in names if n not in exported]
    assert not missing, f"declared but not exported: {missing}"
    for n in names:
        assert hasattr(lib, n)


def test_status_strings(lib):
    for code in range(6):
        assert sas.sas_status_str(code)
    assert sas.sas_status_str(sas.SAS_ERR_TIMEOUT) == "device wait timed out"


@pytest.mark.parametrize("kw,expect", [
    (dict(B=0, H=1, N=128, d=64, topk=2), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=0, d=64, topk=2), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=96, topk=2), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, H=1, N=128, d=64, topk=2, block=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, H=1, N=128, d=64, topk=-1), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=64, topk=65), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, H=1, N=128, d=64, topk=2, mode=7), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=64, topk=2, selector=5), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=64, topk=2, d_sel=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, H=1, N=128, d=64, topk=2, sm_scale=math.nan), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=64, topk=2, sm_scale=-1.0), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=64, topk=2, gate_act=3), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=64, topk=2, gate_act=-1), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=1, N=128, d=64, topk=2, gate_pos=2), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=6, N=128, d=64, topk=2, Hkv=4), sas.SAS_ERR_INVALID_ARG),      # H not a multiple of Hkv
    (dict(B=1, H=2, N=128, d=64, topk=2, Hkv=4), sas.SAS_ERR_INVALID_ARG),      # more KV heads than heads
    (dict(B=1, H=2, N=128, d=64, topk=2, Hkv=-1), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=2, N=128, d=64, topk=2, max_seqs=-1), sas.SAS_ERR_INVALID_ARG),
    (dict(B=2, H=2, N=128, d=64, topk=2, max_seqs=4), sas.SAS_ERR_INVALID_ARG),          # packed needs B = 1
    (dict(B=1, H=2, N=128, d=64, topk=2, max_seqs=4, max_seqlen=129), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=2, N=128, d=64, topk=2, scope=2), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, H=2, N=128, d=64, topk=2, scope=1, gate_pos=1), sas.SAS_ERR_UNSUPPORTED),   # full scope: inner only
    (dict(B=1, H=2, N=128, d=64, topk=2, scope=1, gate_act=1), sas.SAS_ERR_UNSUPPORTED),   # full scope: softmax only
    (dict(B=1, H=2, N=128, d=64, topk=2, scope=1, max_seqs=2), sas.SAS_ERR_UNSUPPORTED),   # full scope: no packing
    (dict(B=1, H=2, N=128, d=64, topk=2, mode=2, scope=1), sas.SAS_ERR_UNSUPPORTED),       # hard-STE: sparse scope
    (dict(B=1, H=2, N=128, d=64, topk=2, mode=2, gate_act=1), sas.SAS_ERR_UNSUPPORTED),    # hard-STE: softmax gates
    (dict(B=1, H=2, N=128, d=64, topk=2, mode=2, gate_pos=1), sas.SAS_ERR_UNSUPPORTED),    # hard-STE: inner position
])
def test_create_rejects_bad_configs(lib, kw, expect):
    assert sas.sas_create_status(**kw) == expect


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU path")
def test_create_without_gpu_fails_cleanly(lib):
    st = sas.sas_create_status(B=1, H=1, N=128, d=64, topk=2)
    assert st in (sas.SAS_ERR_CUDA, sas.SAS_ERR_UNSUPPORTED)


def test_null_handle_and_null_arguments(lib):
    null = ctypes.c_void_p()
    assert lib.sas_attention_fwd(null, *([None] * 10), None) == sas.SAS_ERR_INVALID_ARG
    assert lib.sas_attention_fwd_noisy(null, *([None] * 11), None) == sas.SAS_ERR_INVALID_ARG
    assert lib.sas_mlp_fwd(null, None, None, None, None, None, None, 1, 64, 64, None) == sas.SAS_ERR_INVALID_ARG
    v = ctypes.c_int32()
    assert lib.sas_get_device_status(null, ctypes.byref(v)) == sas.SAS_ERR_INVALID_ARG
    assert lib.sas_launch_count(null) == 0
    lib.sas_destroy(null)   # no-op


def test_binding_refuses_cpu_tensors(lib):
    with pytest.raises(ValueError):
        sas._ptr(torch.zeros(4), torch.float32, "x")


@pytest.mark.parametrize("kw,expect", [
    (dict(B=0, Hq=8, Hkv=2, d=128, topk=4, max_blocks=16, num_pages=32), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, Hq=12, Hkv=8, d=128, topk=4, max_blocks=16, num_pages=32), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, Hq=24, Hkv=8, d=128, topk=4, max_blocks=16, num_pages=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, Hq=8, Hkv=2, d=96, topk=4, max_blocks=16, num_pages=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, Hq=8, Hkv=2, d=128, d_sel=32, topk=4, max_blocks=16, num_pages=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=-1, max_blocks=16, num_pages=32), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=65, max_blocks=16, num_pages=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=4, max_blocks=0, num_pages=32), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=4, max_blocks=40000, num_pages=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=4, max_blocks=16, num_pages=0), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=4, max_blocks=16, num_pages=32, dense=2), sas.SAS_ERR_INVALID_ARG),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=4, max_blocks=16, num_pages=32, block=32), sas.SAS_ERR_UNSUPPORTED),
    (dict(B=1, Hq=8, Hkv=2, d=128, topk=4, max_blocks=16, num_pages=32, sm_scale=math.nan), sas.SAS_ERR_INVALID_ARG),
])
def test_decode_create_rejects_bad_configs(lib, kw, expect):
    assert sas.sas_decode_create_status(**kw) == expect


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU path")
def test_decode_create_without_gpu_fails_cleanly(lib):
    st = sas.sas_decode_create_status(B=1, Hq=8, Hkv=2, d=128, topk=4, max_blocks=16, num_pages=32)
    assert st in (sas.SAS_ERR_CUDA, sas.SAS_ERR_UNSUPPORTED)


def test_decode_null_handle(lib):
    null = ctypes.c_void_p()
    assert lib.sas_decode_step(null, *([None] * 14)) == sas.SAS_ERR_INVALID_ARG
    assert lib.sas_decode_summarize(null, *([None] * 6)) == sas.SAS_ERR_INVALID_ARG
    assert lib.sas_decode_launch_count(null) == 0
