"""The benchmark's algorithmic FLOP counts against a row-by-row count from
the oracle's per-row formula (attention over the kept keys, 4 d per key, plus
the selector's score products): the closed-form block sums of bench.py, the
per-sequence sum of packed layers, and the backward's 10 d per attended pair.
CPU only."""
import bench
from oracle import backward_oracle as BO
from oracle import sas_oracle as O


def _rows(N, K, d, d_sel=0):
    return sum(O.attention_flops_row(i, 64, K, d, d_sel) for i in range(N))


def test_attention_flops_match_the_row_sum():
    for N, K in ((4608, 32), (1000, 4), (129, 0), (64, 32)):
        w = dict(B=2, H=3, N=N, d=128, topk=K, d_sel=128, D=64, F=64)
        f = bench.algorithmic_flops(w, learned=False)
        assert f["attention"] == 2 * 3 * _rows(N, K, 128)
        assert f["selector"] == 0


def test_selector_flops_with_the_learned_selector():
    # per row: 2 d_s C_i score products + 2 d d_s query projection; per full key block 2 d d_s
    N, d, ds = 700, 64, 32
    w = dict(B=1, H=1, N=N, d=d, topk=4, d_sel=ds, D=64, F=64)
    f = bench.algorithmic_flops(w, learned=True)
    rows = sum(2 * ds * (i // 64) + 2 * d * ds for i in range(N))
    assert f["selector"] == rows + (N // 64) * 2 * d * ds


def test_packed_flops_sum_the_sequences():
    w = dict(bench.WORKLOADS["qwen3_4b_packed"])
    f = bench.packed_flops(w)
    assert sum(w["lens"]) == w["N"]
    assert f["attention"] == w["H"] * sum(_rows(n, w["topk"], w["d"]) for n in w["lens"])
    assert f["mlp"] == 4 * w["N"] * w["D"] * w["F"]


def test_backward_flops_are_ten_d_per_attended_pair():
    # the oracle's backward count equals 10/4 of the forward's attention count per head
    N, K, d = 900, 5, 128
    assert BO.backward_flops_head(N, 64, K, d) * 4 == _rows(N, K, d) * 10


def test_training_flops_of_the_three_forms():
    # sparse: 4 d + 10 d per attended pair; full scope: every key j <= i of row i
    # attended (K = C_i); hard-STE: the sparse count plus 4 d per historical key
    N, K, d, B, H = 700, 3, 128, 2, 3
    w = dict(B=B, H=H, N=N, d=d, topk=K, d_sel=128, D=64, F=64)
    fwd, bwd = bench.train_flops(w, "sparse")
    assert fwd == B * H * _rows(N, K, d) and bwd * 4 == fwd * 10
    fwd_f, bwd_f = bench.train_flops(w, "full")
    assert fwd_f == B * H * sum(4 * d * (i + 1) for i in range(N)) and bwd_f * 4 == fwd_f * 10
    fwd_s, bwd_s = bench.train_flops(w, "ste")
    assert fwd_s == fwd
    assert bwd_s - bwd == B * H * sum(4 * d * 64 * (i // 64) for i in range(N))
