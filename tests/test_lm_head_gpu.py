"""Draft logits and candidates through the C ABI (fovea_lm_head_topk) against
the oracle: z = W_LM h_hat (Eq. hidden_correction) and the K_c largest logits
per row, descending, smaller token index first on ties.

Logits are compared with a bound derived from fp32 accumulation of bf16
products; candidate lists match the oracle's exactly except where two
oracle logits lie within that bound of each other (a near-tie), where the
GPU's entry must lie inside the band around the oracle's."""

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fovea():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_22883_gb300 import fovea as f
    f.lib()
    return f


def bf16(x):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)


def check(fovea, V, d, N, k_c, seed, ties=False):
    g = np.random.default_rng(seed)
    W = g.standard_normal((V, d)) / np.sqrt(d)
    h = g.standard_normal((N, d))
    if ties:
        W[V // 2] = W[3]                      # duplicated vocabulary rows tie exactly
        W[V - 1] = W[3]
    Wt, ht = bf16(W).cuda(), bf16(h).cuda()
    W64 = Wt.double().cpu().numpy()
    h64 = ht.double().cpu().numpy()
    ws = fovea.lm_head_workspace(V, d, N, k_c)
    idx, val, logits = fovea.lm_head_topk(Wt, ht, k_c, ws)
    torch.cuda.synchronize()
    fovea.sync_errors(ws)
    ref = oracle.lm_head_topk(W64, h64, k_c)
    z_ref = ref["logits"]
    z = logits.cpu().numpy().astype(np.float64)
    # fp32 accumulation of d exact bf16 products: |error| <= d * 2^-24 * sum |w h|
    bound = d * 2.0 ** -24 * (np.abs(h64) @ np.abs(W64).T) + 1e-30
    assert np.all(np.abs(z - z_ref) <= bound), np.max(np.abs(z - z_ref) / bound)
    idx = idx.cpu().numpy()
    val = val.cpu().numpy().astype(np.float64)
    for n in range(N):
        band = 2 * bound[n].max()
        for r in range(k_c):
            gi, oi = int(idx[n, r]), int(ref["top_idx"][n, r])
            if gi != oi:
                assert abs(z_ref[n, gi] - z_ref[n, oi]) <= band, (n, r, gi, oi)
            assert val[n, r] == np.float32(z[n, gi])
        assert len(set(idx[n].tolist())) == k_c
        assert np.all(np.diff(val[n]) <= 0)
    return idx


@pytest.mark.parametrize("V,d,N,k_c,seed", [
    (1000, 256, 37, 6, 1),       # ragged feature tiles and a ragged row tile
    (777, 320, 5, 32, 2),        # the widest candidate list
    (4099, 192, 130, 1, 3),      # argmax; rows over two row tiles
    (50, 64, 1, 6, 4),           # one row, a vocabulary smaller than a tile
    (2000, 256, 70, 8, 9),       # the widest per-thread candidate list
    (2000, 256, 70, 9, 10),      # the narrowest warp-round list
])
def test_lm_head_topk_matches_oracle(fovea, V, d, N, k_c, seed):
    check(fovea, V, d, N, k_c, seed)


# k_c > 8: one warp per row and K_c warp rounds; k_c <= 8: per-thread lists
@pytest.mark.parametrize("k_c", [32, 9, 8, 6])
def test_lm_head_exact_ties_take_the_smaller_index(fovea, k_c):
    # rows 3, V/2 and V-1 of W_LM are equal: whenever one of them is among the
    # candidates, so are the others in index order (equal logits, equal keys)
    V, d, N = 600, 128, 24
    idx = check(fovea, V, d, N, k_c, 5, ties=True)
    for n in range(N):
        lst = idx[n].tolist()
        pos = [lst.index(j) for j in (3, V // 2, V - 1) if j in lst]
        assert pos == sorted(pos)


# 20 equal rows: a few per thread of a tile's threshold pass; 100: more than
# a thread's list holds in the second tile, so that tile takes the warp rounds
@pytest.mark.parametrize("k_c,block", [(6, 20), (8, 20), (12, 20), (6, 100), (8, 100)])
def test_lm_head_many_equal_largest_logits(fovea, k_c, block):
    """Equal vocabulary rows 246 .. 246 + block - 1, across a 256-column tile
    boundary, hold every row's largest logit: the candidates are the k_c
    smallest of those token indices, in index order, all with one logit."""
    g = np.random.default_rng(11)
    V, d, N = 1000, 128, 33
    W = g.standard_normal((V, d)) / np.sqrt(d)
    W[246:246 + block] = 4.0 / np.sqrt(d)     # far above every other logit for h > 0
    h = np.abs(g.standard_normal((N, d))) + 0.1
    Wt, ht = bf16(W).cuda(), bf16(h).cuda()
    ws = fovea.lm_head_workspace(V, d, N, k_c)
    idx, val, logits = fovea.lm_head_topk(Wt, ht, k_c, ws)
    torch.cuda.synchronize()
    fovea.sync_errors(ws)
    ref = oracle.lm_head_topk(Wt.double().cpu().numpy(), ht.double().cpu().numpy(), k_c)
    want = np.tile(np.arange(246, 246 + k_c, dtype=np.int32), (N, 1))
    assert np.array_equal(ref["top_idx"], want)
    assert np.array_equal(idx.cpu().numpy(), want)
    v = val.cpu().numpy()
    assert np.all(v == v[:, :1])
    assert np.array_equal(v[:, 0], logits.cpu().numpy()[:, 246])


def test_lm_head_vicuna_sized(fovea):
    # a 32000-token vocabulary over d = 4096, 64 draft states, K_c = 6
    check(fovea, 32000, 4096, 64, 6, 6)


def test_lm_head_candidates_without_logits(fovea):
    """logits = NULL: the candidates are those of the call that writes the
    logits, bit for bit."""
    g = np.random.default_rng(8)
    V, d, N, k_c = 3000, 512, 40, 6
    Wt = bf16(g.standard_normal((V, d)) / np.sqrt(d)).cuda()
    ht = bf16(g.standard_normal((N, d))).cuda()
    ws = fovea.lm_head_workspace(V, d, N, k_c)
    idx1, val1, logits = fovea.lm_head_topk(Wt, ht, k_c, ws)
    idx2, val2, none = fovea.lm_head_topk(Wt, ht, k_c, ws, write_logits=False)
    torch.cuda.synchronize()
    fovea.sync_errors(ws)
    assert none is None and logits is not None
    assert torch.equal(idx1, idx2) and torch.equal(val1, val2)
