"""The allocation-free entry point (fovea_retrieve_fuse_noalloc).

Some callers cannot allocate device memory where they run a draft step (a
step recorded into a CUDA graph, a runtime with a fixed memory plan, a loop
that must not pay cudaMalloc's implicit synchronisation).  For them the
library keeps its scratch in a static device array.  This test calls that
entry point through the C ABI, twice in a row on the same array, and checks
each call against fovea_retrieve_fuse with a caller workspace (counts and
indices equal; readout, gate and corrected hidden state within the bf16
tolerance the parity tests use) and against the CPU oracle under the parity
rules.  It checks that the array's error word keeps a device-side condition
until fovea_noalloc_sync_errors reads it, and that a call too large for the
array is refused.  It runs last so a failure here cannot hide other results.
"""

import numpy as np
import pytest
import torch

import workloads
from parity import TOL, compare, params_for, rel_err_rows, run_oracle, store

pytestmark = pytest.mark.gpu


def test_noalloc_entry_point_matches_workspace_entry_point_and_oracle():
    from paper_2608_22883_gb300 import fovea
    w = workloads.generate_custom("noalloc", 512, [300, 77], [40, 9], rho=0.85, k_max=32,
                                  seed=19, temperature=(0.5, 2.0))
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], s.dev.get("mask"))
    ref = fovea.step(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets,
                     s.dev.get("row_scale"), w.rho, w.k_min, w.k_max)
    fovea.sync_errors(ref["workspace"])
    orc, omem = run_oracle(s, mirror=True)
    fovea.noalloc_sync_errors()            # whatever an earlier caller left
    for _ in range(2):
        out = dict(h_out=torch.empty_like(s.dev["h"]),
                   counts=torch.full((w.N,), -7, dtype=torch.int32, device="cuda"),
                   indices=torch.full((w.N, w.k_max), -7, dtype=torch.int32, device="cuda"),
                   readout=torch.empty((w.N, w.d), dtype=torch.float32, device="cuda"),
                   gate=torch.empty(w.N, dtype=torch.float32, device="cuda"))
        fovea.retrieve_fuse_noalloc(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets,
                                    s.dev.get("row_scale"), w.rho, w.k_min, w.k_max, out["h_out"],
                                    counts=out["counts"], indices=out["indices"],
                                    readout=out["readout"], gate=out["gate"])
        fovea.noalloc_sync_errors()
        assert torch.equal(out["counts"], ref["counts"])
        assert torch.equal(out["indices"], ref["indices"])
        tol = TOL[w.dtype]
        for key in ("readout", "h_out"):
            err = rel_err_rows(out[key].double().cpu().numpy(), ref[key].double().cpu().numpy())
            assert err.max() <= tol, (key, err.max())
        assert (out["gate"] - ref["gate"]).abs().max().item() <= tol
        gpu = {k: (v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy())
               for k, v in out.items()}
        compare(gpu, orc, s, mem=omem, mirror=True)
    mem.destroy()


def test_noalloc_error_word_is_kept_until_read():
    from paper_2608_22883_gb300 import fovea
    w = workloads.generate_custom("noalloc-depth", 256, [64], [6], k_max=8, seed=23)
    w.depth = w.depth.copy()
    w.depth[2] = 99                      # outside [0, D]: flagged on the device
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], None)
    h_out = torch.empty_like(s.dev["h"])
    fovea.noalloc_sync_errors()
    fovea.retrieve_fuse_noalloc(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets, None,
                                w.rho, w.k_min, w.k_max, h_out)
    s.dev["depth"][2] = 0
    fovea.retrieve_fuse_noalloc(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets, None,
                                w.rho, w.k_min, w.k_max, h_out)   # a clean call after it
    with pytest.raises(fovea.FoveaError, match="INVALID_ARG"):
        fovea.noalloc_sync_errors()
    fovea.noalloc_sync_errors()          # read and cleared
    mem.destroy()


def test_noalloc_entry_point_refuses_calls_larger_than_its_array():
    from paper_2608_22883_gb300 import fovea
    w = workloads.generate_custom("noalloc-big", 256, [64], [4], k_max=16, seed=5)
    s = store(w)
    params = params_for(s, fovea)
    mem = fovea.build_memory(params, s.dev["v"], None)
    rows = 20000                          # needs far more than the static array
    h = torch.zeros((rows, w.d), dtype=torch.bfloat16, device="cuda")
    depth = torch.zeros(rows, dtype=torch.int32, device="cuda")
    assert fovea.workspace_size(params, mem, [0, rows], 16) > fovea.NOALLOC_WORKSPACE_BYTES
    with pytest.raises(fovea.FoveaError, match="UNSUPPORTED.*static workspace"):
        fovea.retrieve_fuse_noalloc(params, mem, h, depth, [0, rows], None, 0.9, 1, 16,
                                    torch.empty_like(h))
    mem.destroy()
