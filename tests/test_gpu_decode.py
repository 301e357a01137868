"""GPU parity of the SAS decode step (Alg. 2 with per-group selection over a
paged cache) against the fp64 decode oracle, through the C ABI."""
import math

import numpy as np
import pytest
import torch

from oracle import decode_oracle as D
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _append_cpu(K, V, kn, vn, table, lens):
    """The cache the oracle sees: the new token's key and value at position n-1."""
    K, V = K.clone(), V.clone()
    for bi, n in enumerate(lens):
        page = int(table[bi, (n - 1) // 64])
        K[page, :, (n - 1) % 64] = kn[bi]
        V[page, :, (n - 1) % 64] = vn[bi]
    return K, V


def _ulp(x):
    """bf16 spacing at |x| (two steps, so a neighbour across a power of two is covered)."""
    return 2 * np.ldexp(1.0, np.frexp(np.where(x == 0, 2.0 ** -126, x))[1] - 8)


def _rounded_dot_tol(W, x, ref):
    """Bound on |GPU - oracle| for ref = bf16(W @ x): the GPU sums in fp32 (at
    most 2^-17 of sum |W||x| for up to 1024 terms) and both sides round to
    bf16 (one spacing each)."""
    return _ulp(ref) + 2.0 ** -17 * (np.abs(W) @ np.abs(x))


def _score_tol(q_g, Wq_g, K_ctx, Wk, C, d_s):
    """Per-block bound on |s_GPU - s_oracle| from the bounds on q~ and K~."""
    from oracle.sas_oracle import block_summaries, round_to_bf16
    qc = q_g.reshape(-1)
    qt = round_to_bf16(Wq_g @ qc)
    tq = _rounded_dot_tol(Wq_g, qc, qt)
    kbar = block_summaries(K_ctx[:C * 64], 64)
    kt = round_to_bf16(kbar @ Wk.T)
    tk = _ulp(kt) + 2.0 ** -17 * (np.abs(kbar) @ np.abs(Wk).T)
    dot_abs = np.abs(kt) @ np.abs(qt)
    tol = (np.abs(kt) @ tq + tk @ np.abs(qt) + tk @ tq + 2.0 ** -17 * dot_abs) / math.sqrt(d_s)
    return tol, tk


def _check_sets(gpu_sel, ref, K, tol):
    """The GPU's kept set is a valid Top-K of the oracle's scores up to the
    per-block bound tol: no kept block can lie below a dropped one by more
    than their two bounds."""
    s = ref["scores"]
    C = s.shape[0]
    got = gpu_sel[gpu_sel >= 0]
    assert len(got) == min(K, C) and np.all(np.diff(got) > 0)
    if C <= K:
        return True
    if np.array_equal(got, ref["sel"]):
        return True
    out = np.setdiff1d(np.arange(C), got)
    worst_kept = np.argmin(s[got] + tol[got])
    best_dropped = np.argmax(s[out] - tol[out])
    assert s[got][worst_kept] + tol[got][worst_kept] >= s[out][best_dropped] - tol[out][best_dropped], \
        "kept set is not a Top-K even within the rounding bound"
    return False


def run_case(B, Hq, Hkv, d, d_sel, topk, lens, seed=0, exact=False, dense=False, append=True, max_blocks=None,
             groups=None, check_summaries=True):
    G = Hq // Hkv
    max_blocks = max_blocks or max(-(-n // 64) for n in lens) + 1
    table, npages = synth.decode_layout(lens, max_blocks, seed)
    K, V = synth.decode_cache(npages, Hkv, d, seed, device=DEV, exact=exact)
    q, kn, vn = synth.decode_queries(B, Hq, Hkv, d, seed, device=DEV, exact=exact)
    Wq, Wk = synth.decode_selector_weights(Hkv, G, d, d_sel, seed, device=DEV, exact=exact)
    Kcpu, Vcpu = _append_cpu(K.cpu(), V.cpu(), kn.cpu(), vn.cpu(), table, lens)
    if not append:
        K.copy_(Kcpu.to(DEV))
        V.copy_(Vcpu.to(DEV))
    # summaries of blocks nobody wrote stay NaN: reading one would poison the scores
    Ksum = torch.full((B, Hkv, max_blocks, d_sel), float("nan"), device=DEV, dtype=torch.bfloat16)
    dec = sas.SasDecoder(B, Hq, Hkv, d, topk, max_blocks, npages, d_sel=d_sel, dense=dense)
    tab = table.to(DEV)
    lens_t = torch.tensor(lens, dtype=torch.int32, device=DEV)
    if not dense:
        dec.summarize(K, tab, lens_t - 1, Wk, Ksum)
    O, LSE, sel = dec.step(q, K, V, tab, lens_t, kn if append else None, vn if append else None, Wq, Wk,
                           None if dense else Ksum)
    torch.cuda.synchronize()
    assert sas.sas_decode_get_device_status(dec.h) == 0
    launches = sas.sas_decode_launch_count(dec.h)
    dec.close()
    assert torch.equal(K.cpu(), Kcpu) and torch.equal(V.cpu(), Vcpu), "append wrote the wrong cache slots"

    K64 = P.f64(Kcpu)
    ref = D.decode_step(P.f64(q.cpu()), K64, P.f64(Vcpu), table.numpy(), lens, P.f64(Wq.cpu()),
                        P.f64(Wk.cpu()), 64, topk, dense=dense, groups=groups)
    Og, Lg = P.f64(O.cpu()), LSE.cpu().numpy().astype(np.float64)
    sg = None if dense else sel.cpu().numpy()
    Ksum_g = P.f64(Ksum.cpu())
    mism = 0
    q64, Wq64, Wk64 = P.f64(q.cpu()), P.f64(Wq.cpu()), P.f64(Wk.cpu())
    for (bi, g), r in ref["groups"].items():
        hs = slice(g * G, (g + 1) * G)
        if not dense:
            C = r["summaries"].shape[0]
            if not exact and C:
                Kc = D.gather_context(K64, table[bi].numpy(), lens[bi], g, 64)
                tol, tk = _score_tol(q64[bi, hs], Wq64[g], Kc, Wk64[g], C, d_sel)
            if check_summaries and C:
                got = Ksum_g[bi, g, :C]
                if exact:
                    assert np.array_equal(got, r["summaries"]), f"summaries ({bi},{g})"
                else:
                    assert np.all(np.abs(got - r["summaries"]) <= tk), f"summaries ({bi},{g})"
            gs = sg[bi, g, :topk] if topk > 0 else np.zeros(0, dtype=np.int32)
            if exact:
                assert np.array_equal(gs[gs >= 0], r["sel"]), f"sel ({bi},{g})"
                assert np.all(gs[len(r["sel"]):] == -1)
            elif C and not _check_sets(gs, r, topk, tol):
                mism += 1
                continue
        P.compare_o(Og[bi, hs], r["O"], f"O[{bi},{g}]")
        assert np.abs(Lg[bi, hs] - r["LSE"]).max() <= P.LSE_MAX_ABS
    return {"mismatched_groups": mism, "groups": len(ref["groups"]), "launches": launches}


def test_exact_inputs_bit_exact_selection_and_summaries():
    # n = 1 (first token), 65 and 129 (the new token opens a block: the step itself
    # summarises the block it closes), 1000 (ragged current block)
    r = run_case(4, 32, 8, 128, 128, 4, [1, 65, 129, 1000], seed=1, exact=True)
    assert r["launches"] == 4   # summary fill, then the step: prep, selection, attention


def test_random_inputs_qwen_shape_budget_2048():
    r = run_case(3, 32, 8, 128, 128, 32, [4097, 3001, 2200], seed=2)
    assert r["mismatched_groups"] <= 1


@pytest.mark.parametrize("G,d,d_sel,topk", [(1, 64, 64, 3), (2, 128, 64, 0), (8, 64, 128, 5), (4, 128, 128, 64)])
def test_group_sizes_and_dims(G, d, d_sel, topk):
    Hkv = 2
    run_case(2, G * Hkv, Hkv, d, d_sel, topk, [700, 4500], seed=3 + G + topk, exact=True)


def test_dense_decode_matches_oracle():
    run_case(3, 16, 4, 128, 128, 0, [1, 100, 2049], seed=4, dense=True)


def test_dense_long_context_many_splits():
    # 200 blocks per sequence: the dense list is split over many CTAs and merged
    run_case(1, 8, 2, 128, 128, 0, [12800 + 5], seed=5, dense=True, max_blocks=256)


def test_token_already_in_cache():
    run_case(2, 8, 2, 128, 128, 4, [300, 640], seed=6, exact=True, append=False)


def test_keep_all_when_history_short():
    # C <= K for every sequence: every historical block is kept
    run_case(2, 8, 2, 64, 64, 32, [64 * 20 + 3, 64 * 33], seed=7, exact=True)


def test_capacity_larger_than_lengths():
    # grids are sized by the block-table width; most score CTAs find no blocks
    run_case(2, 8, 2, 128, 128, 8, [900, 1500], seed=8, exact=True, max_blocks=4096)


def test_long_context_sampled_groups():
    n = 65536 + 37
    r = run_case(1, 32, 8, 128, 128, 32, [n], seed=9, groups=[(0, 0), (0, 5)], check_summaries=True)
    assert r["mismatched_groups"] == 0


def test_consecutive_steps_in_a_cuda_graph():
    # One captured step replayed while the sequences grow across block
    # boundaries: lengths, queries and the new token are written into the
    # graph's static inputs before every replay.  Summaries of blocks closed
    # during the run come only from the step itself.
    B, Hq, Hkv, d, d_sel, topk = 2, 8, 2, 128, 128, 3
    G = Hq // Hkv
    start = [190, 250]
    steps = 70
    final = [n + steps - 1 for n in start]
    max_blocks = max(-(-n // 64) for n in final) + 1
    table, npages = synth.decode_layout(final, max_blocks, seed=10)
    K, V = synth.decode_cache(npages, Hkv, d, seed=10, device=DEV, exact=True)
    Wq, Wk = synth.decode_selector_weights(Hkv, G, d, d_sel, seed=10, device=DEV, exact=True)
    Ksum = torch.full((B, Hkv, max_blocks, d_sel), float("nan"), device=DEV, dtype=torch.bfloat16)
    tab = table.to(DEV)
    dec = sas.SasDecoder(B, Hq, Hkv, d, topk, max_blocks, npages, d_sel=d_sel)
    dec.summarize(K, tab, torch.tensor([n - 1 for n in start], dtype=torch.int32, device=DEV), Wk, Ksum)
    lens_s = torch.tensor(start, dtype=torch.int32, device=DEV)
    q_s = torch.zeros(B, Hq, d, device=DEV, dtype=torch.bfloat16)
    kn_s = torch.zeros(B, Hkv, d, device=DEV, dtype=torch.bfloat16)
    vn_s = torch.zeros_like(kn_s)
    out = (torch.empty(B, Hq, d, device=DEV, dtype=torch.bfloat16),
           torch.empty(B, Hq, device=DEV, dtype=torch.float32),
           torch.empty(B, Hkv, topk, device=DEV, dtype=torch.int32))
    Kcpu, Vcpu = K.cpu(), V.cpu()
    inputs = [synth.decode_queries(B, Hq, Hkv, d, seed=100 + s, device=DEV, exact=True) for s in range(steps)]
    stream = torch.cuda.Stream()
    # warm-up step outside capture (the same inputs as step 0 are replayed below)
    q_s.copy_(inputs[0][0]); kn_s.copy_(inputs[0][1]); vn_s.copy_(inputs[0][2])
    with torch.cuda.stream(stream):
        dec.step(q_s, K, V, tab, lens_s, kn_s, vn_s, Wq, Wk, Ksum, out=out, stream=stream)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        dec.step(q_s, K, V, tab, lens_s, kn_s, vn_s, Wq, Wk, Ksum, out=out, stream=torch.cuda.current_stream())
    for s in range(steps):
        q, kn, vn = inputs[s]
        lens = [n + s for n in start]
        q_s.copy_(q); kn_s.copy_(kn); vn_s.copy_(vn)
        lens_s.copy_(torch.tensor(lens, dtype=torch.int32))
        graph.replay()
        Kcpu, Vcpu = _append_cpu(Kcpu, Vcpu, kn.cpu(), vn.cpu(), table, lens)
        if s in (0, 2, 5, 66, steps - 1):   # 2 and 66 open new blocks for the two sequences
            torch.cuda.synchronize()
            ref = D.decode_step(P.f64(q.cpu()), P.f64(Kcpu), P.f64(Vcpu), table.numpy(), lens, P.f64(Wq.cpu()),
                                P.f64(Wk.cpu()), 64, topk)
            assert np.array_equal(out[2].cpu().numpy(), ref["sel_idx"]), f"step {s}"
            for bi in range(B):
                P.compare_o(P.f64(out[0][bi].cpu()), ref["O"][bi], f"step {s} O[{bi}]")
                for g in range(Hkv):
                    summ = ref["groups"][(bi, g)]["summaries"]
                    assert np.array_equal(P.f64(Ksum[bi, g, :summ.shape[0]].cpu()), summ)
    torch.cuda.synchronize()
    assert sas.sas_decode_get_device_status(dec.h) == 0
    assert torch.equal(K.cpu(), Kcpu) and torch.equal(V.cpu(), Vcpu)
    dec.close()


def test_repeated_steps_are_identical():
    # the arrival counters return to zero after every launch
    B, Hq, Hkv, d = 2, 16, 4, 128
    lens = [3000, 5000]
    table, npages = synth.decode_layout(lens, 100, seed=11)
    K, V = synth.decode_cache(npages, Hkv, d, seed=11, device=DEV)
    q, _, _ = synth.decode_queries(B, Hq, Hkv, d, seed=11, device=DEV)
    Wq, Wk = synth.decode_selector_weights(Hkv, 4, d, 128, seed=11, device=DEV)
    Ksum = torch.zeros(B, Hkv, 100, 128, device=DEV, dtype=torch.bfloat16)
    dec = sas.SasDecoder(B, Hq, Hkv, d, 16, 100, npages)
    tab, lt = table.to(DEV), torch.tensor(lens, dtype=torch.int32, device=DEV)
    dec.summarize(K, tab, lt, Wk, Ksum)
    outs = [dec.step(q, K, V, tab, lt, Wq=Wq, Wk=Wk, Ksum=Ksum) for _ in range(3)]
    torch.cuda.synchronize()
    assert sas.sas_decode_get_device_status(dec.h) == 0
    dec.close()
    for o in outs[1:]:
        assert all(torch.equal(a, b) for a, b in zip(o, outs[0]))


@pytest.mark.parametrize("bad", ["zero_length", "past_capacity", "missing_page"])
def test_out_of_range_lengths_and_pages_are_reported(bad):
    # Lengths and page indices live on the device: the kernels check them
    # before reading anything, skip the sequence and record INVALID_ARG.
    B, Hq, Hkv, d = 2, 8, 2, 64
    lens = [200, 300]
    table, npages = synth.decode_layout(lens, 8, seed=12)
    K, V = synth.decode_cache(npages, Hkv, d, seed=12, device=DEV)
    q, kn, vn = synth.decode_queries(B, Hq, Hkv, d, seed=12, device=DEV)
    Wq, Wk = synth.decode_selector_weights(Hkv, 4, d, 64, seed=12, device=DEV)
    Ksum = torch.zeros(B, Hkv, 8, 64, device=DEV, dtype=torch.bfloat16)
    if bad == "zero_length":
        lens = [0, 300]
    elif bad == "past_capacity":
        lens = [8 * 64 + 1, 300]
    else:
        table[0, 1] = -1
    dec = sas.SasDecoder(B, Hq, Hkv, d, 2, 8, npages, d_sel=64)
    dec.step(q, K, V, table.to(DEV), torch.tensor(lens, dtype=torch.int32, device=DEV), kn, vn, Wq, Wk, Ksum)
    assert sas.sas_decode_get_device_status(dec.h) == sas.SAS_ERR_INVALID_ARG
    # the context stays usable and the next valid step succeeds
    good, _ = synth.decode_layout([200, 300], 8, seed=12)
    dec.step(q, K, V, good.to(DEV), torch.tensor([200, 300], dtype=torch.int32, device=DEV), kn, vn, Wq, Wk, Ksum)
    assert sas.sas_decode_get_device_status(dec.h) == 0
    dec.close()
