"""Pins of the CPU oracle against things other than itself.

Each check compares the oracle with an independent source: a library routine
of another package (torch.nn.functional, scipy), a closed form, exhaustive
enumeration on tiny inputs, or a hand-derived fixture under tests/golden/.
The mutation tests at the end plant a plausible mistake in a copy of an
oracle function and show that one of the pins catches it.
"""

import dataclasses
import itertools
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

import oracle
from oracle import fovea_oracle as fo
import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "selection_cases.json")


def t64(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float64))


def small_params(d=64, H=32, seed=11):
    p = workloads.draw_params(d, seed, H=H)
    return {k: v.astype(np.float64) for k, v in p.items()}


# ----------------------------------------------------------------------------
# Storage rounding
# ----------------------------------------------------------------------------

def test_round_bf16_matches_torch_on_fp32_values():
    g = np.random.default_rng(0)
    x = np.concatenate([
        g.standard_normal(20000) * 10.0 ** g.integers(-30, 30, 20000),
        g.standard_normal(2000) * 1e-39,                # bf16 subnormals
        np.array([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 3.0e38, -3.3e38, 0.0]),
    ]).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).double().numpy()
    got = oracle.round_bf16(x.astype(np.float64))
    np.testing.assert_array_equal(got, want)


def test_round_bf16_rounds_float64_directly():
    # Closed forms: ties go to even, and a float64 value just above a tie rounds
    # up (rounding through float32 first would land on the tie and go down).
    assert oracle.round_bf16(1 + 2 ** -8) == 1.0
    assert oracle.round_bf16(1 + 3 * 2 ** -8) == 1 + 2 ** -6
    assert oracle.round_bf16(1 + 2 ** -8 + 2 ** -40) == 1 + 2 ** -7
    assert oracle.round_bf16(-(1 + 2 ** -8 + 2 ** -40)) == -(1 + 2 ** -7)
    assert np.isinf(oracle.round_bf16(3.4e38))


# ----------------------------------------------------------------------------
# Elementary operators against torch.nn.functional
# ----------------------------------------------------------------------------

def test_layer_norm_and_rms_norm_match_torch():
    g = np.random.default_rng(1)
    x = g.standard_normal((7, 96)) * 3 + 1.5
    gamma, beta = 1 + 0.1 * g.standard_normal(96), 0.1 * g.standard_normal(96)
    want = F.layer_norm(t64(x), (96,), t64(gamma), t64(beta), eps=1e-5).numpy()
    np.testing.assert_allclose(oracle.layer_norm(x, gamma, beta, 1e-5), want, rtol=1e-12, atol=1e-12)
    want = F.rms_norm(t64(x), (96,), t64(gamma), eps=1e-6).numpy()
    np.testing.assert_allclose(oracle.rms_norm(x, gamma, 1e-6), want, rtol=1e-12, atol=1e-12)


def test_query_matches_torch_linear():
    p = small_params()
    g = np.random.default_rng(2)
    h = g.standard_normal((9, 64))
    depth = np.array([0, 1, 1, 2, 3, 4, 5, 6, 2])
    x = F.layer_norm(t64(h), (64,), t64(p["ln_h_gamma"]), t64(p["ln_h_beta"]), eps=1e-5)
    x = x + t64(p["E_dep"])[torch.as_tensor(depth)]
    want = F.linear(x, t64(p["W_Q"])).numpy()
    np.testing.assert_allclose(oracle.query(p, h, depth), want, rtol=1e-12, atol=1e-12)


def test_memory_matches_torch_with_scattered_mask():
    p = small_params()
    g = np.random.default_rng(3)
    v = g.standard_normal((2, 11, 64))
    mask = (g.random((2, 11)) < 0.6).astype(np.uint8)
    mask[1] = 0
    mask[1, 10] = 1
    mem = oracle.build_memory(p, v, mask)
    for b in range(2):
        valid = np.flatnonzero(mask[b])
        x = F.layer_norm(t64(v[b, valid]), (64,), t64(p["ln_v_gamma"]), t64(p["ln_v_beta"]), eps=1e-5)
        np.testing.assert_array_equal(mem.index[b], valid)
        np.testing.assert_allclose(mem.keys[b], F.linear(x, t64(p["W_K"])).numpy(), rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(mem.values[b], F.linear(x, t64(p["W_U"])).numpy(), rtol=1e-12, atol=1e-12)


def torch_fusion(p, h, r, rms_eps=1e-6):
    """The correction and gate networks as torch modules: two biased linears
    around SiLU each, the gate squashed by a sigmoid, then RMSNorm."""
    d = h.shape[1]
    H = p["b_f1"].shape[0]
    f = torch.nn.Sequential(torch.nn.Linear(2 * d, H), torch.nn.SiLU(), torch.nn.Linear(H, d)).double()
    gnet = torch.nn.Sequential(torch.nn.Linear(2 * d, H), torch.nn.SiLU(), torch.nn.Linear(H, 1)).double()
    with torch.no_grad():
        f[0].weight.copy_(t64(p["W_f1"])); f[0].bias.copy_(t64(p["b_f1"]))
        f[2].weight.copy_(t64(p["W_f2"])); f[2].bias.copy_(t64(p["b_f2"]))
        gnet[0].weight.copy_(t64(p["W_g1"])); gnet[0].bias.copy_(t64(p["b_g1"]))
        gnet[2].weight.copy_(t64(p["w_g2"])[None, :]); gnet[2].bias.copy_(t64(p["b_g2"]))
        z = torch.cat([t64(h), t64(r)], dim=1)
        c = f(z)
        gate = torch.sigmoid(gnet(z))[:, 0]
        y = t64(h) + gate[:, None] * c
        out = F.rms_norm(y, (d,), t64(p["rms_gamma"]), eps=rms_eps)
    return c.numpy(), gate.numpy(), out.numpy()


def test_fusion_matches_torch_modules():
    p = small_params()
    g = np.random.default_rng(4)
    h, r = g.standard_normal((5, 64)), g.standard_normal((5, 64))
    c, gate, out = torch_fusion(p, h, r)
    got = oracle.fuse(p, h, r)
    np.testing.assert_allclose(got["c"], c, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(got["gate"], gate, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(got["h_out"], out, rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------
# Selection: golden fixtures, brute force, closed forms
# ----------------------------------------------------------------------------

def golden_cases():
    with open(GOLDEN) as f:
        return json.load(f)["cases"]


@pytest.mark.parametrize("case", golden_cases(), ids=lambda c: c["name"])
def test_selection_golden(case, select=None, readout=None):
    select = select or oracle.select
    readout = readout or oracle.readout
    p = np.asarray(case["p"], dtype=np.float64)
    s = np.log(p) + case["shift"] if p.size else p
    S = select(s, float(np.float32(case["rho"])), case["k_min"], case["k_max"])
    assert S.K_raw == case["K_raw"]
    assert S.K == case["K"]
    assert list(S.selected) == case["selected"]
    U = np.arange(len(p) * 3, dtype=np.float64).reshape(len(p), 3) ** 1.5
    r, alpha = readout(s, S.selected, U if len(p) else np.zeros((0, 3)))
    np.testing.assert_allclose(alpha, case["alpha"], rtol=1e-12, atol=1e-15)
    want_r = np.asarray(case["alpha"]) @ U[case["selected"]] if case["selected"] else np.zeros(3)
    np.testing.assert_allclose(r, want_r, rtol=1e-12, atol=1e-15)


def brute_force_min_count(alpha_tilde, rho):
    """Smallest k such that SOME k-subset of entries has mass >= rho, and the
    largest mass of a subset of that size (exhaustive enumeration)."""
    V = len(alpha_tilde)
    for k in range(1, V + 1):
        best = max(sum(alpha_tilde[list(c)]) for c in itertools.combinations(range(V), k))
        if best >= rho:
            return k, best
    return V, sum(alpha_tilde)


@pytest.mark.parametrize("seed", range(40))
def test_selection_brute_force(seed, select=None):
    select = select or oracle.select
    g = np.random.default_rng(100 + seed)
    V = int(g.integers(1, 13))
    s = g.standard_normal(V) * g.uniform(0.2, 4.0)
    rho = float(np.float32(g.uniform(0.3, 0.97)))
    alpha_tilde = scipy.special.softmax(s)
    k_star, best = brute_force_min_count(alpha_tilde, rho)
    S = select(s, rho, 1, V)
    assert S.K_raw == k_star
    assert S.K == k_star
    # the selected set attains the largest mass among subsets of its size
    assert abs(alpha_tilde[S.selected].sum() - best) < 1e-12
    # clamps
    assert select(s, rho, 1, max(1, k_star - 1)).K == max(1, k_star - 1)
    assert select(s, rho, V, V).K == V


def check_invariants(S, V, rho, k_min, k_max):
    assert S.K <= k_max and S.K <= V
    assert S.K >= min(k_min, V)
    if V == 0:
        return
    C = S.cum_mass
    if S.K == S.K_raw:
        assert C[S.K - 1] >= rho or S.K == V          # mass reaches rho (or every entry taken)
        if S.K > max(k_min, 1):
            assert C[S.K - 2] < rho                    # minimal count
    if S.K_raw <= k_max and S.K_raw >= k_min and S.K_raw <= V and C[-1] >= rho:
        assert S.K == S.K_raw


@pytest.mark.parametrize("seed", range(20))
def test_selection_invariants(seed):
    g = np.random.default_rng(200 + seed)
    V = int(g.integers(0, 300))
    s = g.standard_normal(V) * g.uniform(0.1, 6.0)
    for rho in (0.5, 0.8, 0.9, 0.99, 1.0):
        rho = float(np.float32(rho))
        for k_min, k_max in ((1, 16), (1, 256), (32, 256), (5, 5)):
            S = oracle.select(s, rho, k_min, k_max)
            check_invariants(S, V, rho, k_min, k_max)
            if V:
                np.testing.assert_allclose(S.alpha_tilde, scipy.special.softmax(s), rtol=1e-12)


def test_one_hot_closed_form():
    g = np.random.default_rng(5)
    s = g.standard_normal(200)
    s[37] = 50.0
    U = g.standard_normal((200, 8))
    S = oracle.select(s, float(np.float32(0.9)), 1, 64)
    assert S.K == 1 and list(S.selected) == [37]
    r, alpha = oracle.readout(s, S.selected, U)
    assert alpha[0] == 1.0
    np.testing.assert_array_equal(r, U[37])


@pytest.mark.parametrize("V,rho", [(10, 0.55), (37, 0.8), (100, 0.333), (64, 0.9)])
def test_uniform_scores_closed_form(V, rho):
    rho = float(np.float32(rho))
    assert abs(rho * V - round(rho * V)) > 1e-3      # rho V not an integer
    s = np.full(V, 0.7)
    U = np.random.default_rng(6).standard_normal((V, 5))
    S = oracle.select(s, rho, 1, V)
    K = math.ceil(rho * V)
    assert S.K_raw == K and S.K == K
    assert list(S.selected) == list(range(K))
    r, _ = oracle.readout(s, S.selected, U)
    np.testing.assert_allclose(r, U[:K].mean(0), rtol=1e-12, atol=1e-14)


def test_dense_case_is_textbook_attention():
    # K_min = K_max = |V| keeps every entry: r = softmax(q K^T / sqrt d) U.
    g = np.random.default_rng(7)
    d, V = 32, 50
    q, K, U = g.standard_normal(d), g.standard_normal((V, d)), g.standard_normal((V, d))
    s = oracle.scores(q, K, d)
    S = oracle.select(s, 1.0, V, V)
    r, _ = oracle.readout(s, S.selected, U)
    want = F.scaled_dot_product_attention(t64(q)[None, None, None], t64(K)[None, None],
                                          t64(U)[None, None])[0, 0, 0].numpy()
    np.testing.assert_allclose(r, want, rtol=1e-12, atol=1e-12)


def test_fixed_top_k_case():
    g = np.random.default_rng(8)
    s = np.round(g.standard_normal(120), 1)          # many exact ties
    K = 16
    S = oracle.select(s, 0.5, K, K)
    want = sorted(range(120), key=lambda i: (-s[i], i))[:K]
    assert list(S.selected) == want
    U = g.standard_normal((120, 4))
    r, alpha = oracle.readout(s, S.selected, U)
    np.testing.assert_allclose(alpha, torch.softmax(t64(s[want]), 0).numpy(), rtol=1e-12)


# ----------------------------------------------------------------------------
# Whole-step identities of the gate (Eq. hidden_correction)
# ----------------------------------------------------------------------------

def small_step(p, seed=9, d=64, M=(20, 7), rows=(5, 3)):
    g = np.random.default_rng(seed)
    v = g.standard_normal((len(M), max(M), d))
    mask = np.zeros((len(M), max(M)), np.uint8)
    for b, m in enumerate(M):
        mask[b, :m] = 1
    h = g.standard_normal((sum(rows), d))
    depth = g.integers(0, 7, sum(rows))
    offs = np.concatenate([[0], np.cumsum(rows)])
    return v, mask, h, depth, offs


def test_zero_gate_returns_rmsnorm_of_h():
    p = small_params()
    p["w_g2"] = np.zeros_like(p["w_g2"])
    p["b_g2"] = np.array([-1000.0])
    v, mask, h, depth, offs = small_step(p)
    mem = oracle.build_memory(p, v, mask)
    out = oracle.retrieve_fuse(p, mem, h, depth, offs, None, 0.9, 1, 8)
    assert np.all(out["gate"] == 0.0)
    want = F.rms_norm(t64(h), (64,), t64(p["rms_gamma"]), eps=1e-6).numpy()
    np.testing.assert_allclose(out["h_out"], want, rtol=1e-12, atol=1e-12)
    # and it no longer depends on the memory values, rho or the correction net
    mem.values = [u * -3.0 + 1.0 for u in mem.values]
    p2 = dict(p, W_f2=p["W_f2"] * 5.0)
    out2 = oracle.retrieve_fuse(p2, mem, h, depth, offs, None, 0.5, 1, 8)
    np.testing.assert_array_equal(out2["h_out"], out["h_out"])


def test_unit_gate_and_zero_correction():
    p = small_params()
    v, mask, h, depth, offs = small_step(p, seed=10)
    mem = oracle.build_memory(p, v, mask)
    p1 = dict(p, w_g2=np.zeros_like(p["w_g2"]), b_g2=np.array([1000.0]))
    out = oracle.retrieve_fuse(p1, mem, h, depth, offs, None, 0.9, 1, 8)
    assert np.all(out["gate"] == 1.0)
    want = F.rms_norm(t64(h + out["c"]), (64,), t64(p["rms_gamma"]), eps=1e-6).numpy()
    np.testing.assert_allclose(out["h_out"], want, rtol=1e-12, atol=1e-12)
    p0 = dict(p, W_f2=np.zeros_like(p["W_f2"]), b_f2=np.zeros_like(p["b_f2"]))
    out0 = oracle.retrieve_fuse(p0, mem, h, depth, offs, None, 0.9, 1, 8)
    want = F.rms_norm(t64(h), (64,), t64(p["rms_gamma"]), eps=1e-6).numpy()
    np.testing.assert_allclose(out0["h_out"], want, rtol=1e-12, atol=1e-12)


def test_depth_gate_leaves_deep_rows_uncorrected():
    """The experimental setup applies the visual correction to nodes of depth
    at most 1: with l_max = 1 a deeper row keeps h_n itself as its scoring
    representation and retrieves nothing, every other row is what the
    ungated step gives, and l_max = D gates nothing."""
    p = small_params()
    v, mask, h, _, offs = small_step(p, seed=21, M=(30, 9), rows=(6, 5))
    depth = np.array([0, 1, 2, 6, 1, 3, 0, 1, 5, 2, 4])
    mem = oracle.build_memory(p, v, mask)
    full = oracle.retrieve_fuse(p, mem, h, depth, offs, None, 0.9, 1, 8)
    gated = oracle.retrieve_fuse(p, mem, h, depth, offs, None, 0.9, 1, 8, l_max=1)
    deep = depth > 1
    np.testing.assert_array_equal(gated["h_out"][deep], h[deep])     # the input itself
    assert np.all(gated["counts"][deep] == 0) and np.all(gated["indices"][deep] == -1)
    assert np.all(gated["gate"][deep] == 0.0) and np.all(gated["readout"][deep] == 0.0)
    np.testing.assert_array_equal(gated["counts"][~deep], full["counts"][~deep])
    np.testing.assert_array_equal(gated["indices"][~deep], full["indices"][~deep])
    for key in ("readout", "h_out", "gate"):
        np.testing.assert_allclose(gated[key][~deep], full[key][~deep], rtol=1e-12, atol=1e-14)
    same = oracle.retrieve_fuse(p, mem, h, depth, offs, None, 0.9, 1, 8, l_max=6)
    np.testing.assert_array_equal(same["indices"], full["indices"])
    np.testing.assert_allclose(same["h_out"], full["h_out"], rtol=1e-12, atol=1e-14)


def test_step_matches_composition_of_torch_pieces():
    """The whole step re-derived with torch ops row by row: query, scores with
    row scale, selection (python sort), softmax over the selected, readout, and
    the torch fusion modules."""
    p = small_params()
    v, mask, h, depth, offs = small_step(p, seed=12, M=(30, 0, 9), rows=(4, 2, 3))
    row_scale = np.random.default_rng(13).uniform(0.2, 3.0, h.shape[0])
    mem = oracle.build_memory(p, v, mask)
    rho, kmin, kmax = float(np.float32(0.8)), 2, 6
    out = oracle.retrieve_fuse(p, mem, h, depth, offs, row_scale, rho, kmin, kmax)
    x = F.layer_norm(t64(h), (64,), t64(p["ln_h_gamma"]), t64(p["ln_h_beta"]), eps=1e-5)
    q = F.linear(x + t64(p["E_dep"])[torch.as_tensor(depth)], t64(p["W_Q"]))
    R = np.zeros_like(h)
    for n in range(h.shape[0]):
        b = int(np.searchsorted(offs, n, side="right") - 1)
        valid = np.flatnonzero(mask[b])
        xv = F.layer_norm(t64(v[b, valid]), (64,), t64(p["ln_v_gamma"]), t64(p["ln_v_beta"]), eps=1e-5)
        Kb, Ub = F.linear(xv, t64(p["W_K"])), F.linear(xv, t64(p["W_U"]))
        s = (Kb @ q[n]) / 8.0 * row_scale[n]
        V = len(valid)
        if V == 0:
            assert out["counts"][n] == 0 and np.all(out["indices"][n] == -1)
            continue
        at = torch.softmax(s, 0).numpy()
        order = sorted(range(V), key=lambda i: (-float(s[i]), i))
        cum, k_raw = 0.0, V
        for k, i in enumerate(order, 1):
            cum += at[i]
            if cum >= rho:
                k_raw = k
                break
        K = min(V, kmax, max(kmin, k_raw))
        sel = order[:K]
        assert out["counts"][n] == K
        assert list(out["indices"][n, :K]) == list(valid[sel])
        w = torch.softmax(s[sel], 0)
        R[n] = (w[:, None] * Ub[sel]).sum(0).numpy()
    np.testing.assert_allclose(out["readout"], R, rtol=1e-10, atol=1e-12)
    _, _, want = torch_fusion(p, h, R)
    np.testing.assert_allclose(out["h_out"], want, rtol=1e-10, atol=1e-12)


# ----------------------------------------------------------------------------
# Mirror rounding and the planted workload
# ----------------------------------------------------------------------------

def test_mirror_rounds_at_the_storage_points():
    p = small_params()
    v, mask, h, depth, offs = small_step(p, seed=14)
    mem = oracle.build_memory(p, v, mask, mirror=True)
    for k in mem.keys + mem.values:
        np.testing.assert_array_equal(k, oracle.round_bf16(k))
    out = oracle.retrieve_fuse(p, mem, h, depth, offs, None, 0.9, 1, 8, mirror=True)
    for key in ("a_f", "a_g", "h_out"):
        np.testing.assert_array_equal(out[key], oracle.round_bf16(out[key]))
    # q = W_Q x_h is kept exact; x_h = LN(h) + E_dep is rounded
    x = oracle.round_bf16(oracle.layer_norm(h, p["ln_h_gamma"], p["ln_h_beta"], 1e-5) + p["E_dep"][depth])
    np.testing.assert_allclose(out["q"], x @ p["W_Q"].T, rtol=1e-12, atol=1e-12)
    pure = oracle.retrieve_fuse(p, oracle.build_memory(p, v, mask), h, depth, offs, None, 0.9, 1, 8)
    rel = np.abs(out["h_out"] - pure["h_out"]).max() / np.abs(pure["h_out"]).max()
    assert rel < 5e-2


def test_folded_scores_equal_query_scores():
    """Query folding: x . (W_Q^T k) against (W_Q x) . k with q formed by
    torch.nn.functional.linear and the keys by the oracle's build."""
    p = small_params()
    v, mask, h, depth, offs = small_step(p, seed=15)
    mem = oracle.fold_keys(p, oracle.build_memory(p, v, mask))
    x = oracle.query_input(p, h, depth)
    q = F.linear(t64(x), t64(p["W_Q"])).numpy()
    for b in range(len(mem.keys)):
        for n in range(offs[b], offs[b + 1]):
            want = mem.keys[b] @ q[n] / 8.0
            np.testing.assert_allclose(oracle.scores(x[n], mem.folded[b], 64), want,
                                       rtol=1e-11, atol=1e-11)


def test_folded_step_equals_plain_step_in_exact_arithmetic():
    p = small_params()
    v, mask, h, depth, offs = small_step(p, seed=16, M=(30, 0, 9), rows=(4, 2, 3))
    row_scale = np.random.default_rng(17).uniform(0.2, 3.0, h.shape[0])
    mem = oracle.build_memory(p, v, mask)
    a = oracle.retrieve_fuse(p, mem, h, depth, offs, row_scale, 0.8, 2, 6)
    b = oracle.retrieve_fuse(p, mem, h, depth, offs, row_scale, 0.8, 2, 6, fold=True)
    np.testing.assert_array_equal(a["counts"], b["counts"])
    np.testing.assert_array_equal(a["indices"], b["indices"])
    for key in ("readout", "h_out", "gate"):
        np.testing.assert_allclose(b[key], a[key], rtol=1e-10, atol=1e-12)


def test_folded_mirror_rounds_the_folded_keys():
    p = small_params()
    v, mask, h, depth, offs = small_step(p, seed=18)
    mem = oracle.build_memory(p, v, mask, mirror=True)
    exact = oracle.fold_keys(p, mem)
    fm = oracle.fold_keys(p, mem, mirror=True)
    for kf, ke in zip(fm.folded, exact.folded):
        np.testing.assert_array_equal(kf, oracle.round_bf16(kf))
        assert np.all(np.abs(kf - ke) <= 2.0 ** -8 * np.abs(ke) + 1e-300)   # half a bf16 ulp
    out = oracle.retrieve_fuse(p, fm, h, depth, offs, None, 0.9, 1, 8, mirror=True, fold=True)
    x = oracle.round_bf16(oracle.layer_norm(h, p["ln_h_gamma"], p["ln_h_beta"], 1e-5) + p["E_dep"][depth])
    for n in range(offs[1]):
        np.testing.assert_allclose(out["scores"][n], fm.folded[0] @ x[n] / 8.0, rtol=1e-12, atol=1e-12)


def test_planted_rows_are_peaked():
    spec = workloads.Spec(0, "planted-small", d=256, B=1, rows_per_seq=12, rho=0.9,
                          k_max=16, k_min=1, dtype="fp32", seed=21, m_fixed=96,
                          peaked_rows=4)
    w = workloads.generate(spec)
    p = {k: a.astype(np.float64) for k, a in w.params.items()}
    mem = oracle.build_memory(p, w.v, w.mask)
    q = oracle.query(p, w.h, w.depth)
    out = oracle.retrieve_fuse(p, mem, w.h, w.depth, w.row_offsets, None, w.rho, 1, 16)
    for row, entry in w.planted.items():
        k = mem.keys[0][entry]
        cos = q[row] @ k / np.linalg.norm(q[row]) / np.linalg.norm(k)
        assert abs(cos - 0.9) < 0.01
        assert out["counts"][row] == 1 and out["indices"][row, 0] == entry
    flat = [n for n in range(w.N) if n not in w.planted]
    assert np.mean(out["counts"][flat]) > 4


def test_workload_draws_are_deterministic():
    a = workloads.generate_custom("t", 64, [10, 3], [4, 2], seed=3, temperature=(0.1, 10))
    b = workloads.generate_custom("t", 64, [10, 3], [4, 2], seed=3, temperature=(0.1, 10))
    for name in workloads.PARAM_NAMES:
        np.testing.assert_array_equal(a.params[name], b.params[name])
    np.testing.assert_array_equal(a.h, b.h)
    np.testing.assert_array_equal(a.row_scale, b.row_scale)
    assert list(a.depth) == [0, 1, 1, 1, 0, 1]
    assert list(workloads.tree_depths(13)) == [0, 1, 1, 1, 1, 1, 1, 2, 3, 4, 5, 6, 2]


# ----------------------------------------------------------------------------
# Mutation checks: a planted mistake is caught by one of the pins above
# ----------------------------------------------------------------------------

def _mutant_select_strict(s, rho, k_min, k_max):
    S = fo.select(s, rho, k_min, k_max)
    if S.K_raw and S.cum_mass[S.K_raw - 1] == rho:        # '>' instead of '>='
        K_raw = S.K_raw + 1
        K = min(len(s), k_max, max(k_min, K_raw))
        return fo.Selection(K, K_raw, S.order, S.cum_mass, S.alpha_tilde, S.order[:K])
    return S


def _mutant_select_tie_last(s, rho, k_min, k_max):
    S = fo.select(s, rho, k_min, k_max)
    V = len(s)
    order = np.lexsort((-np.arange(V), -np.asarray(s)))   # ties: larger index first
    return fo.Selection(S.K, S.K_raw, order, S.cum_mass, S.alpha_tilde, order[:S.K])


def _mutant_readout_global_softmax(s, selected, U):
    if len(selected) == 0:
        return np.zeros(U.shape[1]), np.zeros(0)
    ex = np.exp(np.asarray(s) - np.max(s))
    alpha = (ex / ex.sum())[selected]                     # renormalisation dropped
    return alpha @ U[selected], alpha


@pytest.mark.parametrize("mutant", [
    dict(select=_mutant_select_strict),
    dict(select=_mutant_select_tie_last),
    dict(readout=_mutant_readout_global_softmax),
], ids=["strict-inequality", "tie-order", "no-renormalisation"])
def test_pins_catch_planted_selection_mistakes(mutant):
    failures = 0
    for case in golden_cases():
        try:
            test_selection_golden(case, **mutant)
        except AssertionError:
            failures += 1
    assert failures > 0


def test_pins_catch_transposed_query_and_swapped_concat():
    p = small_params()
    g = np.random.default_rng(2)
    h = g.standard_normal((9, 64))
    depth = np.zeros(9, np.int64)
    bad = dict(p, W_Q=p["W_Q"].T)
    x = F.layer_norm(t64(h), (64,), t64(p["ln_h_gamma"]), t64(p["ln_h_beta"]), eps=1e-5)
    want = F.linear(x + t64(p["E_dep"])[0], t64(p["W_Q"])).numpy()
    assert not np.allclose(oracle.query(bad, h, depth), want, rtol=1e-6)
    r = g.standard_normal((9, 64))
    _, _, want = torch_fusion(p, h, r)
    swapped = oracle.fuse(p, r, h)["h_out"]               # [r; h] instead of [h; r]
    assert not np.allclose(swapped, want, rtol=1e-6)


def test_pins_catch_a_transposed_fold():
    p = small_params()
    v, mask, h, depth, offs = small_step(p, seed=15)
    mem = oracle.build_memory(p, v, mask)
    bad = dataclasses.replace(mem, folded=[K @ p["W_Q"].T for K in mem.keys])   # W_Q k, not W_Q^T k
    x = oracle.query_input(p, h, depth)
    q = F.linear(t64(x), t64(p["W_Q"])).numpy()
    n = 0
    assert not np.allclose(oracle.scores(x[n], bad.folded[0], 64), mem.keys[0] @ q[n] / 8.0,
                           rtol=1e-6)


# ----------------------------------------------------------------------------
# Draft logits and candidates (z = W_LM h_hat, top K_c)
# ----------------------------------------------------------------------------

def test_lm_head_logits_by_explicit_sums():
    g = np.random.default_rng(40)
    V, d, N = 23, 12, 4
    W, h = g.standard_normal((V, d)), g.standard_normal((N, d))
    out = oracle.lm_head_topk(W, h, 5)
    for n in range(N):
        for j in range(V):
            want = math.fsum(W[j, i] * h[n, i] for i in range(d))
            assert abs(out["logits"][n, j] - want) <= 1e-12 * max(1.0, abs(want))


def test_lm_head_topk_brute_force_with_ties():
    g = np.random.default_rng(41)
    V, d, N, k = 40, 8, 6, 6
    W = np.round(g.standard_normal((V, d)), 0)        # integer weights: exact ties
    W[7] = W[3]                                       # duplicated rows tie exactly
    W[30] = W[3]
    h = np.round(g.standard_normal((N, d)) * 2.0, 0)
    h[0] = 0.0                                        # every logit 0: indices 0..k-1
    out = oracle.lm_head_topk(W, h, k)
    for n in range(N):
        z = [sum(W[j, i] * h[n, i] for i in range(d)) for j in range(V)]
        want = sorted(range(V), key=lambda j: (-z[j], j))[:k]
        assert list(out["top_idx"][n]) == want
        assert list(out["top_val"][n]) == [z[j] for j in want]
    assert list(out["top_idx"][0]) == list(range(k))


def test_lm_head_one_hot_rows_closed_form():
    # W_LM[j] = c_j e_{p(j)}: z_{n,j} = c_j h_{n,p(j)}
    g = np.random.default_rng(42)
    V, d = 16, 16
    p = g.permutation(d)
    c = np.arange(1, V + 1, dtype=np.float64)
    W = np.zeros((V, d))
    W[np.arange(V), p] = c
    h = np.ones((1, d))
    out = oracle.lm_head_topk(W, h, 3)
    assert list(out["top_idx"][0]) == [15, 14, 13]
    assert list(out["top_val"][0]) == [16.0, 15.0, 14.0]
