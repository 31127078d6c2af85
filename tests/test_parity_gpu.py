"""GPU parity: the C-ABI path against the CPU oracle on the same stored inputs.

Small cases span several 128-row tiles, ragged tails, masks, empty and single
entry memories, the selection clamps (k_max = 1, k_max > |V|, the paper's
rho = 0.8 / K_min = 32 / K_max = 256, fixed top-16, dense), per-row
temperatures, clustered keys, the depth gate and the fp32 path.  The five
named workloads run at full size (the long-memory one on every row of four of
its hundred steps).

The oracle is always the paper's order of operations: q = W_Q (LN(h) + E_dep)
scored against the keys.  The default bf16 step scores x = LN(h) + E_dep
against the memory's folded keys W_Q^T k (a hi / lo pair), and is held to the
same oracle.
"""

import dataclasses

import numpy as np
import pytest
import torch

import oracle
import workloads
from parity import (LN_EPS, RMS_EPS, compare, params_for, rel_err_rows, run_gpu, run_oracle,
                    store)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fovea():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_22883_gb300 import fovea as f
    f.lib()          # raises if the library was not built: no fallback
    return f


SMALL = {
    "bf16-ragged": dict(d=256, m_sizes=[200, 37, 129], rows=[37, 5, 20], rho=0.9, k_max=16),
    "bf16-scattered-mask-d320": dict(d=320, m_sizes=[150, 90], rows=[13, 40], M_max=220,
                                     scattered_mask=True, rho=0.8, k_max=32),
    "bf16-empty-and-single": dict(d=256, m_sizes=[0, 1, 70], rows=[3, 4, 9], M_max=80, k_max=8),
    "bf16-kmax-1": dict(d=256, m_sizes=[300], rows=[33], k_max=1),
    # one score group, after a sequence without rows: its keys start at entry 120
    "bf16-one-group-offset": dict(d=256, m_sizes=[120, 64], rows=[0, 19], k_max=16),
    "bf16-kmax-beyond-valid": dict(d=256, m_sizes=[45, 3], rows=[10, 6], k_max=256, rho=0.99),
    "bf16-paper-defaults": dict(d=384, m_sizes=[600], rows=[40], rho=0.8, k_min=32, k_max=256),
    "bf16-fixed-top16": dict(d=256, m_sizes=[400, 250], rows=[20, 20], k_min=16, k_max=16),
    "bf16-dense": dict(d=256, m_sizes=[180], rows=[21], k_min=180, k_max=180),
    # dense beyond 256 selected entries: the general selection (bitonic order),
    # the readout kernel and the first fusion layer as a GEMM
    "bf16-dense-wide": dict(d=256, m_sizes=[600], rows=[20], rho=1.0, k_min=600, k_max=600),
    "bf16-temperature": dict(d=512, m_sizes=[256, 1024, 700], rows=[32, 32, 17],
                             temperature=(0.1, 10.0), rho=0.8, k_max=128),
    "bf16-clustered": dict(d=256, m_sizes=[2048], rows=[128], clusters=16, cluster_sigma=0.2,
                           k_max=256),
    "bf16-many-rows": dict(d=256, m_sizes=[130, 500], rows=[300, 4], k_max=64),
    # more rows than twice the SMs: the selection writes dense weights and one
    # GEMM against the transposed projected values forms the first fusion layer
    "bf16-many-rows-dense-weights": dict(d=256, m_sizes=[130, 500, 77], rows=[300, 10, 40],
                                         k_max=64, temperature=(0.3, 3.0)),
    # rows beyond 2048 entries: selection and readout run as two kernels
    "bf16-long-rows": dict(d=256, m_sizes=[2500, 300], rows=[12, 5], k_max=64),
    "bf16-hidden-128": dict(d=256, m_sizes=[100], rows=[9], k_max=16, H=128),
    # fewer entries than d: the memory holds folded keys; clustered near-ties
    "bf16-clustered-folded": dict(d=1024, m_sizes=[768], rows=[96], clusters=16,
                                  cluster_sigma=0.2, k_max=128),
    # caps above 256 with the mass rule deciding K: candidates put in order by
    # the bucket order, the mass scanned four entries per thread (rows of up to
    # 2048 entries, and beyond)
    "bf16-large-cap": dict(d=256, m_sizes=[1500, 700], rows=[16, 8], rho=0.95, k_max=512,
                           temperature=(0.25, 1.2)),
    "bf16-long-rows-large-cap": dict(d=256, m_sizes=[3000], rows=[10], rho=0.9, k_max=400,
                                     temperature=(0.25, 1.2)),
    "fp32-large-cap": dict(d=128, m_sizes=[900], rows=[6], dtype="fp32", rho=0.9, k_max=300,
                           temperature=(0.25, 1.2)),
    "fp32-ragged": dict(d=256, m_sizes=[64, 130], rows=[4, 11], dtype="fp32", k_max=16),
    "fp32-temperature": dict(d=192, m_sizes=[300, 20], rows=[17, 3], dtype="fp32", k_max=64,
                             temperature=(0.1, 10.0), rho=0.8),
}


def small_workload(name):
    kw = dict(SMALL[name])
    return workloads.generate_custom(name, kw.pop("d"), kw.pop("m_sizes"), kw.pop("rows"), **kw)


# Boundary-row share allowed per small case (at least three rows; the
# boundary rows follow from the oracle alone, so the counts are fixed per
# seeded case): clustered keys cut between near-equal scores, temperatures
# up to 10 widen the score scale, and the paper's defaults with K_min = 32
# sit near the mass threshold on a few rows.
SMALL_MAX_EXEMPT = {"bf16-clustered": 0.1, "bf16-temperature": 0.1, "bf16-paper-defaults": 0.1,
                    # flat rows with K in the hundreds: one entry moves the mass by
                    # ~1e-3, so the 1e-4 band catches about a quarter of them
                    "bf16-large-cap": 0.35, "bf16-long-rows-large-cap": 0.3}


@pytest.mark.parametrize("name", sorted(SMALL))
def test_small_parity(fovea, name):
    w = small_workload(name)
    s = store(w)
    gpu = run_gpu(s, fovea)
    orc, mem = run_oracle(s, mirror=(w.dtype == "bf16"))
    rep = compare(gpu, orc, s, mem=mem, mirror=(w.dtype == "bf16"),
                  max_exempt=SMALL_MAX_EXEMPT.get(name, 0.05))
    print(f"{name} (folded: {gpu['_folded']}): boundary rows {rep['exempt']}, readout err {rep['readout_err']:.2e}, "
          f"h_out err {rep['h_out_err']:.2e}, gate err {rep['gate_err']:.2e}")


@pytest.mark.parametrize("name", ["bf16-ragged", "bf16-scattered-mask-d320", "fp32-ragged",
                                  "bf16-empty-and-single"])
def test_memory_build_matches_oracle(fovea, name):
    w = small_workload(name)
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], s.dev.get("mask"))
    K, U, idx, offs = mem.views()
    orc = oracle.build_memory({n: s.f64[n] for n in workloads.PARAM_NAMES}, s.f64["v"],
                              s.f64.get("mask"), mirror=(w.dtype == "bf16"))
    assert mem.valid_counts == [len(i) for i in orc.index]
    idx = idx.cpu().numpy()
    tol = 2e-2 if w.dtype == "bf16" else 1e-4
    kappa = mem.folded_keys(params)
    assert (kappa is not None) == (w.dtype == "bf16" and mem.total > 0)
    if kappa is not None:
        # the exact fold of the (bf16) keys: the GPU keeps it as hi + lo
        orc = oracle.fold_keys({n: s.f64[n] for n in workloads.PARAM_NAMES}, orc, mirror=False)
        kappa = kappa.double().cpu().numpy()
        kappa = kappa[:, :w.d] + kappa[:, w.d:]
    for b in range(w.B):
        lo, hi = offs[b], offs[b + 1]
        np.testing.assert_array_equal(idx[lo:hi], orc.index[b])
        if hi == lo:
            continue
        for got, ref in [(K, orc.keys[b]), (U, orc.values[b])]:
            g = got[lo:hi].double().cpu().numpy()
            assert rel_err_rows(g, ref).max() <= tol
            if w.dtype == "bf16":
                assert np.mean(g == ref) > 0.99     # same bf16 value almost everywhere
        if kappa is not None:
            # about 16 significant bits plus the fp32 accumulation of W_Q^T k
            assert rel_err_rows(kappa[lo:hi], orc.folded[b]).max() <= 2e-4
    mem.destroy()


def test_plain_fusion_when_weights_differ(fovea):
    """The memory keeps the values projected through the r-half of the first
    fusion layer for the W_f1 / W_g1 it was built with.  A bf16 call given
    other W_f1 / W_g1 pointers (here copies holding the same values) takes the
    plain path: the readout r, then the first fusion layer as a GEMM over
    [h; r].  Both paths match the oracle, and each other within the bf16
    tolerance, with identical selections."""
    w = small_workload("bf16-ragged")
    s = store(w)
    params = params_for(s, fovea)
    fovea.timing_enable(True)
    proj = run_gpu(s, fovea, params=params)
    names_proj = set(fovea.timing_read())
    orc, mem = run_oracle(s, mirror=True)
    weights = {n: s.dev[n] for n in workloads.PARAM_NAMES}
    weights["W_f1"] = weights["W_f1"].clone()
    weights["W_g1"] = weights["W_g1"].clone()
    other = fovea.Params(weights, d_model=w.d, mlp_hidden=w.params["b_f1"].shape[0],
                         max_depth=w.params["E_dep"].shape[0] - 1, dtype=fovea.BF16)
    fovea.timing_enable(True)              # clears the records
    plain = run_gpu(s, fovea, params=other, memory=proj["_memory"])
    names_plain = set(fovea.timing_read())
    fovea.timing_enable(False)
    assert "select_fuse" in names_proj and "fuse_hidden" not in names_proj
    assert "fuse_hidden" in names_plain and "select_fuse" not in names_plain
    assert proj["_folded"] == plain["_folded"]           # same W_Q: the same score form
    for gpu in (proj, plain):
        compare(gpu, orc, s, mem=mem, mirror=True)
    np.testing.assert_array_equal(proj["counts"], plain["counts"])
    np.testing.assert_array_equal(proj["indices"], plain["indices"])
    assert rel_err_rows(proj["h_out"].astype(np.float64), plain["h_out"].astype(np.float64)).max() <= 2e-2


@pytest.mark.parametrize("name", ["bf16-clustered-folded", "bf16-scattered-mask-d320",
                                  "bf16-one-group-offset"])
def test_folded_and_unfolded_steps_select_the_same_entries(fovea, name):
    """A memory built without W_Q holds no folded keys: the step then forms
    q = W_Q x_h (hi / lo pair) and scores it against the keys, the paper's
    own order.  A memory built with W_Q scores x_h against the folded keys
    (hi / lo pair).  Both match the paper-order oracle, and both give the
    same counts and the same ordered index lists on every row outside the
    boundary band."""
    w = small_workload(name)
    s = store(w)
    params = params_for(s, fovea)
    no_wq = {n: s.dev[n] for n in workloads.PARAM_NAMES if n != "W_Q"}
    build_params = fovea.Params(no_wq, d_model=w.d, mlp_hidden=w.params["b_f1"].shape[0],
                                max_depth=w.params["E_dep"].shape[0] - 1, dtype=fovea.BF16)
    plain_mem = fovea.build_memory(build_params, s.dev["v"], s.dev.get("mask"))
    assert plain_mem.folded_keys(params) is None
    fovea.timing_enable(True)
    plain = run_gpu(s, fovea, params=params, memory=plain_mem)
    names_plain = set(fovea.timing_read())
    fovea.timing_enable(True)
    folded = run_gpu(s, fovea, params=params)
    names_folded = set(fovea.timing_read())
    fovea.timing_enable(False)
    assert not plain["_folded"] and folded["_folded"]
    assert "query_proj" in names_plain and not any(n.startswith("score_f") for n in names_plain)
    assert "query_proj" not in names_folded
    assert any(n in names_folded for n in ("score_folded", "score_fusion_h"))
    orc, mem = run_oracle(s, mirror=True)
    cap = SMALL_MAX_EXEMPT.get(name, 0.05)
    rp = compare(plain, orc, s, mem=mem, mirror=True, max_exempt=cap)
    rf = compare(folded, orc, s, mem=mem, mirror=True, max_exempt=cap)
    same = [n for n in range(w.N) if n not in rp["exempt"]]
    np.testing.assert_array_equal(plain["counts"][same], folded["counts"][same])
    for n in same:
        assert sorted(plain["indices"][n]) == sorted(folded["indices"][n]), f"row {n}: sets differ"
    # the order inside a list may differ only between near-equal scores (both
    # lists passed the oracle's order check above)
    differ = [n for n in range(w.N) if set(plain["indices"][n]) != set(folded["indices"][n])]
    reordered = [n for n in range(w.N) if n not in differ
                 and not np.array_equal(plain["indices"][n], folded["indices"][n])]
    print(f"{name}: rows whose selected sets differ between the folded and unfolded steps: "
          f"{differ} (boundary rows {sorted(rp['exempt'])}); same set, near-tie order swapped: "
          f"{len(reordered)}")


def test_paths_are_taken(fovea):
    """bf16 rows of up to 2048 entries, caps of up to 256 and batches of up
    to twice the SMs run the selection, the projected readout and the first
    fusion layer's activation in one kernel; otherwise the selection writes
    dense weights and one GEMM against the transposed projected values forms
    the activation (the readout, when asked for, has its own kernel); fp32
    takes the unfolded SIMT path with the first fusion layer as a GEMM."""
    try:
        for name, want, absent in (
                # several score groups: G_h in a launch of its own
                ("bf16-ragged",
                 {"ln_query", "fusion_h", "score_folded", "select_fuse", "fuse_out", "finalize"},
                 "query_proj"),
                ("bf16-one-group-offset", {"score_fusion_h", "select_fuse"}, "score_folded"),
                # long rows: selection with dense weights, the weighted sum as a GEMM
                ("bf16-long-rows", {"score_folded", "select", "readout", "act_gemm", "fuse_out"},
                 "fuse_hidden"),
                ("bf16-many-rows-dense-weights", {"select", "act_gemm"}, "select_fuse"),
                ("bf16-dense-wide", {"select", "act_gemm"}, "fuse_hidden"),
                ("fp32-ragged", {"query_proj", "score", "select_readout", "fuse_hidden"},
                 "select_fuse")):
            s = store(small_workload(name))
            fovea.timing_enable(True)
            run_gpu(s, fovea)
            names = set(fovea.timing_read())
            fovea.timing_enable(False)
            assert want <= names and absent not in names, (name, names)
    finally:
        fovea.timing_enable(False)


@pytest.mark.parametrize("name", ["bf16-ragged", "bf16-long-rows", "fp32-ragged"])
def test_depth_gate(fovea, name):
    """l_max = 1 (the experimental setup corrects nodes of depth <= 1): a
    deeper row keeps h (bit for bit), count 0, indices -1, gate 0, readout 0;
    the other rows match the oracle.  Runs the projected path, the path of
    rows beyond 2048 entries, and fp32."""
    w = small_workload(name)
    s = store(w)
    gpu = run_gpu(s, fovea, l_max=1)
    orc, mem = run_oracle(s, mirror=(w.dtype == "bf16"), l_max=1)
    assert orc["gated"].sum() > 0 and (~orc["gated"]).sum() > 0
    compare(gpu, orc, s, mem=mem, mirror=(w.dtype == "bf16"))
    assert np.all(gpu["readout"][orc["gated"]] == 0.0)


def test_zero_gate_returns_rmsnorm_of_h(fovea):
    w = small_workload("bf16-ragged")
    w.params["w_g2"] = np.zeros_like(w.params["w_g2"])
    w.params["b_g2"] = np.array([-1000.0], dtype=np.float32)
    s = store(w)
    gpu = run_gpu(s, fovea)
    assert np.all(gpu["gate"] == 0.0)
    h = s.f64["h"]
    want = oracle.round_bf16(oracle.rms_norm(h, s.f64["rms_gamma"], 1e-6))
    assert rel_err_rows(gpu["h_out"].astype(np.float64), want).max() <= 2e-2


def test_planted_rows_select_one_entry(fovea):
    spec = workloads.Spec(0, "planted-d512", d=512, B=1, rows_per_seq=24, rho=0.9, k_max=32,
                          k_min=1, dtype="bf16", seed=31, m_fixed=300, peaked_rows=6)
    w = workloads.generate(spec)
    s = store(w)
    gpu = run_gpu(s, fovea)
    for row, entry in w.planted.items():
        assert gpu["counts"][row] == 1 and gpu["indices"][row, 0] == entry
    orc, mem = run_oracle(s, mirror=True)
    compare(gpu, orc, s, mem=mem)


def test_repeat_calls_are_deterministic(fovea):
    w = small_workload("bf16-temperature")
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], s.dev.get("mask"))
    ws = fovea.new_workspace(params, mem, w.row_offsets, w.k_max)
    outs = []
    for _ in range(3):
        o = fovea.step(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets,
                       s.dev.get("row_scale"), w.rho, w.k_min, w.k_max, workspace=ws)
        torch.cuda.synchronize()
        outs.append({k: v.clone() for k, v in o.items() if k != "workspace" and v is not None})
    for o in outs[1:]:
        for k in o:
            assert torch.equal(o[k], outs[0][k]), k
    fovea.sync_errors(ws)


def test_invalid_depth_sets_error_word(fovea):
    w = small_workload("bf16-ragged")
    w.depth = w.depth.copy()
    w.depth[3] = 9
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], s.dev.get("mask"))
    o = fovea.step(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets, None, w.rho, 1, 16)
    with pytest.raises(fovea.FoveaError, match="INVALID_ARG"):
        fovea.sync_errors(o["workspace"])
    fovea.sync_errors(o["workspace"])      # the word was cleared


def test_bounded_wait_that_gives_up_reports_timeout(fovea):
    """Every mbarrier wait of the tensor-core kernels is bounded.  With the
    limit cut to 1 ns (fovea_debug_wait_limit) the waits give up while the
    copies and MMAs they wait for are still in flight: each kernel records
    FOVEA_ERR_TIMEOUT, waits for the work it issued with its fixed limits,
    and exits.  The call's status reads TIMEOUT through fovea_sync_errors,
    which clears the workspace header; after fovea_workspace_init the same
    workspace serves a normal call that matches the oracle."""
    w = small_workload("bf16-temperature")
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], s.dev.get("mask"))
    ws = fovea.new_workspace(params, mem, w.row_offsets, w.k_max)
    fovea.debug_wait_limit(1)
    try:
        fovea.step(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets,
                   s.dev.get("row_scale"), w.rho, w.k_min, w.k_max, workspace=ws)
        with pytest.raises(fovea.FoveaError, match="TIMEOUT"):
            fovea.sync_errors(ws)
    finally:
        fovea.debug_wait_limit(0)
    fovea.lib().fovea_workspace_init(ws.data_ptr(), ws.numel(), None)
    out = fovea.step(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets,
                     s.dev.get("row_scale"), w.rho, w.k_min, w.k_max, workspace=ws)
    fovea.sync_errors(ws)
    gpu = {k: (v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy())
           for k, v in out.items() if v is not None and k != "workspace"}
    orc, omem = run_oracle(s, mirror=True)
    compare(gpu, orc, s, mem=omem, max_exempt=SMALL_MAX_EXEMPT["bf16-temperature"])


def test_bad_row_offsets_and_workspace(fovea):
    w = small_workload("bf16-ragged")
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], s.dev.get("mask"))
    ws = fovea.new_workspace(params, mem, w.row_offsets, 16)
    h_out = torch.empty_like(s.dev["h"])
    for offs in ([1, 37, 42, 62], [0, 37, 20, 62]):
        with pytest.raises(fovea.FoveaError, match="INVALID_ARG"):
            fovea.retrieve_fuse(params, mem, s.dev["h"], s.dev["depth"], offs, None, 0.9, 1, 16,
                                h_out, ws)
    with pytest.raises(fovea.FoveaError, match="INVALID_ARG"):
        fovea.retrieve_fuse(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets, None, 0.9, 1,
                            16, h_out, ws[:1024])
    with pytest.raises(fovea.FoveaError, match="UNSUPPORTED"):
        fovea.retrieve_fuse(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets, None, 0.9, 1,
                            4096, h_out, ws)
    # zero draft states: nothing to do
    fovea.retrieve_fuse(params, mem, s.dev["h"], s.dev["depth"], [0, 0, 0, 0], None, 0.9, 1, 16,
                        h_out, ws)
    fovea.sync_errors(ws)


# ---------------------------------------------------------------------------
# The five named workloads at full size
# ---------------------------------------------------------------------------

# Boundary-row share allowed per named workload.  In the long-memory one every
# row reaches the 256 cap, and its clustered keys put 11-13 % of those cuts
# between scores within the tie band.
NAMED_MAX_EXEMPT = {1: 0.05, 2: 0.05, 3: 0.05, 4: 0.05, 5: 0.15}


@pytest.mark.parametrize("idx", [1, 2, 3, 4])
def test_named_workload_parity(fovea, idx):
    w = workloads.generate(workloads.WORKLOADS[idx])
    s = store(w)
    gpu = run_gpu(s, fovea)
    orc, mem = run_oracle(s, mirror=(w.dtype == "bf16"))
    rep = compare(gpu, orc, s, mem=mem, mirror=(w.dtype == "bf16"),
                  max_exempt=NAMED_MAX_EXEMPT[idx])
    print(f"workload {idx} (folded keys: {gpu['_folded']}): {rep['rows']} rows, boundary rows "
          f"{len(rep['exempt'])} ({rep['exempt_mass']} mass, {rep['exempt_tie']} tie; GPU selection "
          f"differs from the oracle's on {rep['exempt_differ']}) {rep['exempt']}, readout err "
          f"{rep['readout_err']:.2e}, h_out err {rep['h_out_err']:.2e}, gate err {rep['gate_err']:.2e}")
    if idx == 2:
        for row, entry in w.planted.items():
            assert gpu["counts"][row] == 1 and gpu["indices"][row, 0] == entry
        assert (gpu["counts"] == w.k_max).sum() > 16        # flat rows reach the cap
    if idx == 3:
        assert gpu["counts"].min() == 1 and gpu["counts"].max() == w.k_max


def test_long_memory_steps(fovea):
    """Long-memory workload: one memory of 4 x 8192 clustered entries queried
    over 100 draft steps.  The GPU runs every step; the oracle checks every
    row of every sequence at steps 0, 1, 49 and 99."""
    spec = workloads.WORKLOADS[5]
    w0 = workloads.generate(spec, step=0)
    s0 = store(w0)
    params = params_for(s0, fovea)
    mem = fovea.build_memory(params, s0.dev["v"], s0.dev.get("mask"))
    ws = fovea.new_workspace(params, mem, w0.row_offsets, w0.k_max)
    p64 = {n: s0.f64[n] for n in workloads.PARAM_NAMES}
    omem = oracle.build_memory(p64, s0.f64["v"], None, mirror=True, ln_eps=LN_EPS)
    checked = {}
    for t in range(spec.steps):
        h = workloads.hidden_states(spec.seed, w0.N, spec.d, step=t)
        ht = torch.from_numpy(h).to(torch.bfloat16).cuda()
        out = fovea.step(params, mem, ht, s0.dev["depth"], w0.row_offsets, None, w0.rho,
                         w0.k_min, w0.k_max, workspace=ws)
        if t not in (0, 1, 49, 99):
            continue
        torch.cuda.synchronize()
        gpu = {k: (v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy())
               for k, v in out.items() if v is not None and k != "workspace"}
        ws_t = store(dataclasses.replace(w0, h=h), device=None)
        orc = oracle.retrieve_fuse(p64, omem, ws_t.f64["h"], ws_t.f64["depth"], w0.row_offsets,
                                   None, w0.rho, w0.k_min, w0.k_max, mirror=True,
                                   ln_eps=LN_EPS, rms_eps=RMS_EPS)
        rep = compare(gpu, orc, ws_t, mem=omem, mirror=True, max_exempt=NAMED_MAX_EXEMPT[5])
        checked[t] = (len(rep["exempt"]), rep["exempt_mass"], rep["exempt_tie"],
                      len(rep["exempt_differ"]), rep["readout_err"], rep["h_out_err"])
    fovea.sync_errors(ws)
    assert sorted(checked) == [0, 1, 49, 99]
    print("long memory, step: (boundary rows, mass, tie, boundary rows whose GPU selection "
          f"differs, readout err, h_out err) of {w0.N} rows: {checked}")
