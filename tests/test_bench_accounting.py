"""The bench's algorithmic byte and flop accounting (the roofline numerators)
against figures fixed independently of it: the per-step upper bound of the
LLaVA-7B-shaped workload (65.1 MB, 3.83 GFLOP with every row selecting
K_max distinct entries, capped by the memory size), and the terms each
restatement removes (query folding: W_Q and the query GEMM; projected
values: the r-half of the first fusion layer and the d-wide value rows)."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workloads  # noqa: E402


@pytest.fixture(scope="module")
def w7b():
    return workloads.generate(workloads.WORKLOADS[2])


def upper_bound_selection(w):
    """Every row selects K_max entries; the union of a sequence's rows covers
    min(M, R K_max) distinct entries (here all of them)."""
    N, K = w.N, w.k_max
    counts = np.full(N, K, np.int64)
    idx = np.tile(np.arange(K), (N, 1))
    for n in range(N):
        idx[n] = (np.arange(K) + n * K) % int(w.m_sizes[0])
    return counts, idx


def test_method_bytes_and_flops_match_the_upper_bound(w7b):
    counts, idx = upper_bound_selection(w7b)
    nbytes, flops, uniq = bench.step_cost(w7b, counts, idx, False)
    assert uniq == 576
    assert abs(nbytes / 1e6 - 65.1) < 0.15            # W_Q 33.6 + fusion 21.0 + K 4.7 + U 4.7 + io 1.05
    assert abs(flops / 1e9 - 3.83) < 0.02


def test_folding_and_projection_remove_their_terms(w7b):
    counts, idx = upper_bound_selection(w7b)
    d, H, N = w7b.d, int(w7b.params["b_f1"].shape[0]), w7b.N
    plain, f_plain, uniq = bench.step_cost(w7b, counts, idx, False)
    proj, f_proj, _ = bench.step_cost(w7b, counts, idx, True)
    both, f_both, _ = bench.step_cost(w7b, counts, idx, True, True)
    # projected values: the r-half of [W_f1 ; W_g1] (2H x d) no longer read,
    # value rows 2H wide instead of d wide
    assert plain - proj == 2 * (2 * H * d) + 2 * uniq * (d - 2 * H)
    # folding: W_Q (d x d, bf16) no longer read, no query GEMM; the folded
    # keys are a hi / lo pair, twice the key bytes
    M = int(w7b.m_sizes[0])
    assert proj - both == 2 * d * d - 2 * M * d
    assert f_proj - f_both == 2 * N * d * d
    assert abs(both / 1e6 - 24.3) < 0.1


def test_kernel_bytes_of_the_folded_launches(w7b):
    d, H, N, M = w7b.d, int(w7b.params["b_f1"].shape[0]), w7b.N, int(w7b.m_sizes[0])
    merged = bench.kernel_bytes("score_fusion_h", w7b, 0, True)
    # folded keys (hi, lo) + the h-halves of W_f1, W_g1 + x_h and h (bf16); scores and G_h out (fp32)
    assert merged == (2 * M * d + 2 * H * d + 2 * N * d) * 2 + N * M * 4 + N * 2 * H * 4
    # the two separate launches (several score groups) move the same bytes:
    # x_h in the one, h in the other
    assert bench.kernel_bytes("score_folded", w7b, 0, True) + bench.kernel_bytes("fusion_h", w7b, 0, True) \
        == merged


def test_kernel_bytes_of_the_dense_weights_launches():
    """Long-memory shape (4 images of 8192 entries, 512 rows, 2H = 1024):
    the selection writes the weights as a bf16 hi / lo pair [512, 8192]
    (16.8 MB), and the activation GEMM reads them with the transposed
    projected values [4, 1024, 8192] (67.1 MB) and G_h, writing the
    activations."""
    w = workloads.WORKLOADS[5]
    class W:                                     # the shape alone; no inputs drawn
        d, N, B, k_max = w.d, w.N, w.B, w.k_max
        m_sizes = [8192] * 4
        row_offsets = [0, 128, 256, 384, 512]
        dtype = "bf16"
        params = {"b_f1": np.zeros(512)}
    alpha = 512 * 8192 * 2 * 2
    projT = 4 * 1024 * 8192 * 2
    assert bench.kernel_bytes("select", W, 0, True, True) - bench.kernel_bytes("select", W, 0, True) == alpha
    act = bench.kernel_bytes("act_gemm", W, 0, True, True)
    assert act == alpha + projT + 2 * 1024 + 512 * 1024 * 2 + 512 * 1024 * 4
    assert abs(act / 1e6 - 87.0) < 0.1         # 16.8 + 67.1 + 1.0 (act out) + 2.1 (G_h in)
