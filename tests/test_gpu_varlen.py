"""GPU parity of the packed variable-length forward (cu_seqlens offsets on the
device; each sequence its own causal problem with its own block partition)
against the fp64 oracle, bit-identity with the batched path on equal
lengths, and device-side rejection of bad offsets (status word, no fault)."""
import numpy as np
import pytest
import torch

from oracle import sas_oracle as OR
from paper_2609_13141_gb300 import sas, synth
from tests import parity as P

pytestmark = pytest.mark.gpu

TRAIN, INFER = sas.SAS_MODE_TRAIN_SOFT, sas.SAS_MODE_INFER_HARD
DEV = torch.device("cuda:0")


def _packed(lens, cap, Hq, Hkv, d, max_len, seed):
    Q = synth.qkv(1, Hq, cap, d, seed=seed)[0][0]
    _, K, V = synth.qkv(1, Hkv, cap, d, seed=seed + 100)
    S = synth.scores(1, Hkv, cap, -(-max_len // 64), seed=seed, regime="R1")[0]
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32)
    return Q, K[0], V[0], S, cu


def _run(lens, cap, Hq, Hkv, d, topk, mode, max_len, Q, K, V, S, cu):
    layer = sas.SasLayer(1, Hq, cap, d, topk, mode=mode, Hkv=Hkv, max_seqs=max(len(lens), 1), max_seqlen=max_len)
    O, LSE, si, sl = layer.attention_varlen(cu.to(DEV), *(t.to(DEV).contiguous() for t in (Q, K, V, S)),
                                            sel_fill=-7)   # a value the library never writes
    status = sas.sas_get_device_status(layer.h)
    layer.close()
    return {"O": O.cpu(), "LSE": LSE.cpu(), "sel_idx": si.cpu(), "sel_logg": sl.cpu(), "status": status}


@pytest.mark.parametrize("lens,cap,Hq,Hkv,d,topk,mode", [
    ([700, 1, 64, 129, 0, 300, 255], 1500, 4, 2, 128, 3, TRAIN),   # ragged, empty, one-token, GQA, spare rows
    ([513, 130, 77], 720, 2, 2, 64, 2, INFER),                     # d = 64, inference form, offsets off the block grid
    ([300, 17, 140, 1], 500, 8, 1, 128, 3, TRAIN),                 # G = 8: head-packed tiles of 16 tokens
])
def test_varlen_matches_oracle(lens, cap, Hq, Hkv, d, topk, mode):
    max_len = max(lens)
    Q, K, V, S, cu = _packed(lens, cap, Hq, Hkv, d, max_len, seed=len(lens))
    g = _run(lens, cap, Hq, Hkv, d, topk, mode, max_len, Q, K, V, S, cu)
    assert g["status"] == 0
    ref = OR.sas_attention_varlen(P.f64(Q), P.f64(K), P.f64(V), cu.numpy(), 64, topk, P.f64(S), mode=mode)
    end = int(cu[-1])
    rows = np.arange(end)
    for hi in range(Hq):
        P.compare_o(P.f64(g["O"][hi])[:end], ref["O"][hi, :end], f"O[{hi}]")
        assert np.abs(g["LSE"][hi].numpy()[:end] - ref["LSE"][hi, :end]).max() <= P.LSE_MAX_ABS
    for gk in range(Hkv):
        assert np.array_equal(g["sel_idx"][gk].numpy()[:end, :topk], ref["sel_idx"][gk, :end])
        assert np.abs(g["sel_logg"][gk].numpy()[:end, :topk] - ref["sel_logg"][gk, :end]).max() <= P.LOGG_MAX_ABS
    # rows past the last sequence are not written
    assert torch.count_nonzero(g["O"][:, end:]) == 0
    assert bool((g["sel_idx"][:, end:] == -7).all())


def test_equal_lengths_are_bit_identical_to_the_batched_path():
    S_, n, H, d, topk = 3, 700, 4, 128, 4
    Q, K, V, S, cu = _packed([n] * S_, S_ * n, H, H, d, n, seed=9)
    g = _run([n] * S_, S_ * n, H, H, d, topk, TRAIN, n, Q, K, V, S, cu)
    # the same data as a [B = 3, H, n, d] batch
    bat = lambda x: x.reshape(x.shape[0], S_, n, -1).transpose(0, 1).contiguous()
    layer = sas.SasLayer(S_, H, n, d, topk)
    O, LSE, si, sl = layer.attention(*(bat(t).to(DEV) for t in (Q, K, V)), scores=bat(S).to(DEV))
    layer.close()
    unb = lambda x: x.cpu().transpose(0, 1).reshape(x.shape[1], S_ * n, -1)
    assert torch.equal(g["O"], unb(O))
    assert torch.equal(g["LSE"], unb(LSE[..., None])[..., 0])
    assert torch.equal(g["sel_idx"], unb(si))
    assert torch.equal(g["sel_logg"], unb(sl))


def test_long_gqa_pack_sampled_rows():
    lens = [8192, 3000, 64, 5000, 1]
    cap, Hq, Hkv, d, topk = 16384, 8, 2, 128, 32
    Q, K, V, S, cu = _packed(lens, cap, Hq, Hkv, d, 8192, seed=21)
    g = _run(lens, cap, Hq, Hkv, d, topk, TRAIN, 8192, Q, K, V, S, cu)
    assert g["status"] == 0
    # sampled rows of sequences 0 and 3 for query heads 1 and 6
    for s_, hi in ((0, 1), (3, 6)):
        b0, n = int(cu[s_]), lens[s_]
        rows = P.sample_rows(n, 96, seed=s_)
        gk = hi // (Hq // Hkv)
        r = OR.sas_attention_head(P.f64(Q[hi, b0:b0 + n]), P.f64(K[gk, b0:b0 + n]), P.f64(V[gk, b0:b0 + n]),
                                  P.f64(S[gk, b0:b0 + n]), 64, topk, rows=rows)
        P.compare_o(P.f64(g["O"][hi, b0 + rows]), r["O"], f"O[{hi}]")
        assert np.abs(g["LSE"][hi, b0 + rows].numpy() - r["LSE"]).max() <= P.LSE_MAX_ABS
        assert np.array_equal(g["sel_idx"][gk, b0 + rows].numpy()[:, :topk], r["sel_idx"])


def test_bad_offsets_set_the_status_and_compute_nothing():
    lens = [100, 200]
    Q, K, V, S, cu = _packed(lens, 400, 2, 2, 128, 256, seed=4)
    bad = torch.tensor([0, 250, 200], dtype=torch.int32)     # decreasing
    g = _run(lens, 400, 2, 2, 128, 2, TRAIN, 256, Q, K, V, S, bad)
    assert g["status"] == sas.SAS_ERR_INVALID_ARG
    assert torch.count_nonzero(g["O"]) == 0
    too_long = torch.tensor([0, 300, 310], dtype=torch.int32)  # a sequence longer than max_seqlen
    g = _run(lens, 400, 2, 2, 128, 2, TRAIN, 256, Q, K, V, S, too_long)
    assert g["status"] == sas.SAS_ERR_INVALID_ARG
    assert torch.count_nonzero(g["O"]) == 0


def test_wrong_entry_points_are_refused():
    layer = sas.SasLayer(1, 2, 256, 128, 2, max_seqs=2)
    z = torch.zeros(1, 2, 256, 128, device=DEV, dtype=torch.bfloat16)
    with pytest.raises(sas.SasError):
        layer.attention(z, z, z, scores=torch.zeros(1, 2, 256, 4, device=DEV))
    layer.close()
    layer = sas.SasLayer(1, 2, 256, 128, 2)
    with pytest.raises(sas.SasError):
        layer.attention_varlen(torch.tensor([0, 256], dtype=torch.int32, device=DEV), z[0], z[0], z[0],
                               torch.zeros(2, 256, 4, device=DEV))
    layer.close()


@pytest.mark.parametrize("lens,cap,Hq,Hkv,d,topk,mode", [
    ([700, 1, 64, 129, 0, 300, 255], 1500, 4, 2, 128, 3, TRAIN),   # ragged, empty, one-token, GQA, spare rows
    ([513, 130, 77], 720, 2, 2, 64, 2, INFER),                     # d = 64, offsets off the block grid
])
def test_varlen_learned_selector_exact_inputs(lens, cap, Hq, Hkv, d, topk, mode):
    # integer Q, K and {-1, 0, 1} projections: every selector sum is exact in
    # fp32, so each sequence's kept sets -- scored against the summaries of its
    # own blocks with its group gate query -- equal the oracle's on every row
    G = Hq // Hkv
    Q = synth.integer_selector_inputs(1, Hq, cap, d, d, seed=len(lens))[0][0]
    _, K, V, _, _ = synth.integer_selector_inputs(1, Hkv, cap, d, d, seed=len(lens) + 1)
    K, V = K[0], V[0]
    Wq, Wk = synth.decode_selector_weights(Hkv, G, d, d, seed=len(lens), exact=True)
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32)
    max_len = max(lens)
    layer = sas.SasLayer(1, Hq, cap, d, topk, mode=mode, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d, Hkv=Hkv,
                         max_seqs=len(lens), max_seqlen=max_len)
    O, LSE, si, sl = layer.attention_varlen(cu.to(DEV), *(t.to(DEV).contiguous() for t in (Q, K, V)), None,
                                            sel_fill=-7, Wq=Wq.to(DEV), Wk=Wk.to(DEV))
    assert sas.sas_get_device_status(layer.h) == 0
    layer.close()
    ref = OR.sas_attention_varlen(P.f64(Q), P.f64(K), P.f64(V), cu.numpy(), 64, topk, mode=mode, Wq=P.f64(Wq),
                                  Wk=P.f64(Wk))
    end = int(cu[-1])
    for gk in range(Hkv):
        for s0, s1 in zip(cu[:-1].tolist(), cu[1:].tolist()):
            if s1 == s0:
                continue
            s = OR.selector_scores_group(P.f64(Q[gk * G:(gk + 1) * G, s0:s1]), P.f64(K[gk, s0:s1]), P.f64(Wq[gk]),
                                         P.f64(Wk[gk]), 64)
            P.check_selection_rows(si[gk, s0:s1].cpu().numpy()[:, :topk], s, np.arange(s1 - s0), topk)
        assert np.abs(sl[gk].cpu().numpy()[:end, :topk] - ref["sel_logg"][gk, :end]).max() <= P.LOGG_MAX_ABS
    for hi in range(Hq):
        P.compare_o(P.f64(O[hi].cpu())[:end], ref["O"][hi, :end], f"O[{hi}]")
        assert np.abs(LSE[hi].cpu().numpy()[:end] - ref["LSE"][hi, :end]).max() <= P.LSE_MAX_ABS
    assert torch.count_nonzero(O[:, end:]) == 0
    assert bool((si[:, end:] == -7).all())


def test_varlen_learned_equal_lengths_match_the_batched_path():
    # three sequences of 640 tokens packed = a batch of three 640-token sequences
    S_, n, H, d, topk = 3, 640, 2, 128, 4
    Q, K, V = synth.qkv(S_, H, n, d, seed=12, regime="R2")
    Wq, Wk = synth.selector_weights(H, d, d, seed=12)
    dev = DEV
    batched = sas.SasLayer(S_, H, n, d, topk, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d)
    Ob, Lb, sib, slb = batched.attention(*(t.to(dev) for t in (Q, K, V)), Wq=Wq.to(dev), Wk=Wk.to(dev))
    batched.close()
    packed = sas.SasLayer(1, H, S_ * n, d, topk, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=d, max_seqs=S_,
                          max_seqlen=n)
    pack = lambda t: t.permute(1, 0, 2, 3).reshape(t.shape[1], S_ * n, d).contiguous().to(dev)
    cu = torch.arange(0, S_ * n + 1, n, dtype=torch.int32, device=dev)
    Op, Lp, sip, slp = packed.attention_varlen(cu, pack(Q), pack(K), pack(V), None, Wq=Wq.to(dev), Wk=Wk.to(dev))
    assert sas.sas_get_device_status(packed.h) == 0
    packed.close()
    for b in range(S_):
        rows = slice(b * n, (b + 1) * n)
        assert torch.equal(Op[:, rows], Ob[b])
        assert torch.equal(Lp[:, rows], Lb[b])
        assert torch.equal(sip[:, rows], sib[b])
        assert torch.equal(slp[:, rows], slb[b])
