"""Shared parity machinery: store a workload in its dtype, run the C-ABI path
and the CPU oracle on the same stored inputs, and compare them under the
exactness / tolerance rules.

Rules (exact where the path decides an integer, bounded where it rounds, with
the boundary exemption spelled out):
* counts and selected index sets are bit-exact, except rows where the
  oracle's cumulative mass at the decision lies within 1e-4 of rho, or where
  the cut falls inside a score tie band (K-th and (K+1)-th scores within
  1e-4 * max(1, |s_K|)).  Such rows are listed and checked separately: the GPU
  count is within 1 of the oracle's, every entry the GPU and the oracle
  disagree on lies inside the tie band of the cut, and r / h_hat agree with the
  oracle re-evaluated on the GPU's selected set.
* r (readout) and h_hat: per-row max relative error
  ||x_gpu - x_ref||_inf / max(||x_ref||_inf, 1e-30) <= 2e-2 for bf16 and
  <= 1e-4 for fp32.
The order inside a selected list is compared up to swaps of entries whose
scores lie within the same tie band.

The oracle is always the paper-order form (q = W_Q x against the keys), also
for GPU steps that score against the memory's folded keys: the folded keys
carry kappa = W_Q^T k as a hi / lo pair, so both forms agree with q . k to
within fp32 accumulation, far inside the boundary band.

Boundary rows are reported by kind ("mass": the mass reading; "tie": the tie
reading of the cut), and a caller bounds their share (``max_exempt``), so a
band that swallows many rows fails instead of passing silently.
"""

from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional

import numpy as np
import torch

import oracle
import workloads

BAND = 1e-4
TOL = {"bf16": 2e-2, "fp32": 1e-4}
# The gate g = sigma(a_g . w_g2 + b_g2) lies in (0, 1); its absolute error
# comes from the bf16 activations a_g (one ulp flips of single elements move
# the sum by ~1e-4) and from the projected readout's fp32 sum.
GATE_TOL = {"bf16": 5e-3, "fp32": 1e-5}
# The library receives its epsilons as fp32; the oracle uses the same values.
LN_EPS = float(np.float32(1e-5))
RMS_EPS = float(np.float32(1e-6))


def storage_dtype(dtype: str) -> torch.dtype:
    return torch.bfloat16 if dtype == "bf16" else torch.float32


@dataclasses.dataclass
class Stored:
    """A workload's inputs stored in its dtype on the device, and the exact
    stored values as float64 for the oracle."""
    w: workloads.Workload
    dev: Dict[str, torch.Tensor]
    f64: Dict[str, np.ndarray]


def store(w: workloads.Workload, device: str = "cuda", h: Optional[np.ndarray] = None) -> Stored:
    dt = storage_dtype(w.dtype)
    dev, f64 = {}, {}

    def put(name, arr, dtype=dt):
        t = torch.from_numpy(np.ascontiguousarray(arr)).to(dtype)
        dev[name] = t.to(device) if device else t
        f64[name] = t.to(torch.float64).numpy() if t.is_floating_point() else t.numpy()

    for name, arr in w.params.items():
        put(name, arr)
    put("v", w.v)
    put("h", w.h if h is None else h)
    put("depth", w.depth, torch.int32)
    if w.mask is not None:
        put("mask", w.mask, torch.uint8)
    if w.row_scale is not None:
        put("row_scale", w.row_scale, torch.float32)
    return Stored(w, dev, f64)


def params_for(s: Stored, fovea, H=None, D=None):
    w = s.w
    H = H if H is not None else w.params["b_f1"].shape[0]
    D = D if D is not None else w.params["E_dep"].shape[0] - 1
    weights = {n: s.dev[n] for n in workloads.PARAM_NAMES}
    return fovea.Params(weights, d_model=w.d, mlp_hidden=H, max_depth=D,
                        dtype=fovea.BF16 if w.dtype == "bf16" else fovea.FP32)


def oracle_params(s: Stored) -> Dict[str, np.ndarray]:
    return {n: s.f64[n] for n in workloads.PARAM_NAMES}


@dataclasses.dataclass
class RowReport:
    n: int
    exempt: bool
    reason: str


def classify_rows(orc: dict, w: workloads.Workload, rows) -> Dict[int, str]:
    """Rows whose decision sits on a boundary: the cumulative mass lies within
    BAND of rho at K_raw (or K_raw - 1) and moving K_raw by one would change the
    clamped count K ("mass"), or the cut falls inside a score tie band
    ("cut-tie": the order of equal scores is a reading, so a cut between
    near-equal scores decides nothing the paper fixes).  Rows past the depth
    gate have no selection and are never boundary rows."""
    rho = float(np.float32(w.rho))
    out = {}
    for n in rows:
        S = orc["selections"][n]
        if S is None or len(S.order) == 0:
            continue
        C, s = S.cum_mass, orc["scores"][n]
        V = len(S.order)

        def clamp(k_raw):
            return min(V, w.k_max, max(w.k_min, k_raw))

        reasons = []
        kr = S.K_raw
        up = abs(C[kr - 1] - rho) < BAND and clamp(kr + 1) != clamp(kr)
        down = kr >= 2 and abs(C[kr - 2] - rho) < BAND and clamp(kr - 1) != clamp(kr)
        if up or down:
            reasons.append("mass")
        K = S.K
        if K < V:
            sk, sk1 = s[S.order[K - 1]], s[S.order[K]]
            if abs(sk - sk1) < BAND * max(1.0, abs(sk)):
                reasons.append("cut-tie")
        if reasons:
            out[n] = "+".join(reasons)
    return out


def rel_err_rows(x: np.ndarray, ref: np.ndarray) -> np.ndarray:
    num = np.abs(x - ref).max(axis=1)
    den = np.maximum(np.abs(ref).max(axis=1), 1e-30)
    return num / den


def compare(gpu: Dict[str, np.ndarray], orc: dict, s: Stored, rows=None,
            mem: Optional[oracle.Memory] = None, mirror: bool = True,
            max_exempt: float = 0.05) -> dict:
    """Assert parity of GPU outputs with the oracle on `rows` (default: all).
    At most a `max_exempt` share of the rows may be boundary rows.  Returns a
    summary dict (exempt rows by kind, max errors)."""
    w = s.w
    N = w.N
    rows = list(range(N)) if rows is None else list(rows)
    tol = TOL[w.dtype]
    exempt = classify_rows(orc, w, rows)
    n_mass = sum(1 for r in exempt.values() if "mass" in r)
    n_tie = sum(1 for r in exempt.values() if "cut-tie" in r)
    assert len(exempt) <= max(3, max_exempt * len(rows)), \
        f"{len(exempt)} boundary rows of {len(rows)} ({n_mass} mass, {n_tie} tie) exceed {max_exempt:.0%}"
    p = oracle_params(s)
    ref_r = orc["readout"].copy()
    ref_h = orc["h_out"].copy()
    ref_g = orc["gate"].copy()
    gated = orc.get("gated")
    differ = []                  # boundary rows whose GPU selection is not the oracle's
    for n in rows:
        if gated is not None and gated[n]:
            # past the depth gate: not corrected, bit for bit
            assert int(gpu["counts"][n]) == 0, f"gated row {n}: count {gpu['counts'][n]}"
            assert np.all(gpu["indices"][n] == -1), f"gated row {n}: indices set"
            assert np.array_equal(gpu["h_out"][n].astype(np.float64), s.f64["h"][n]), \
                f"gated row {n}: h_out differs from h"
            assert gpu["gate"][n] == 0.0
            continue
        K_o = int(orc["counts"][n])
        K_g = int(gpu["counts"][n])
        idx_g = [int(x) for x in gpu["indices"][n, :K_g]]
        assert all(x == -1 for x in gpu["indices"][n, K_g:]), f"row {n}: indices not -1 padded"
        S = orc["selections"][n]
        if n not in exempt:
            assert K_g == K_o, f"row {n}: count {K_g} != oracle {K_o}"
            idx_o = [int(x) for x in orc["indices"][n, :K_o]]
            assert sorted(idx_g) == sorted(idx_o), f"row {n}: selected sets differ"
            if K_o:
                _check_order(orc, w, mem, n, idx_g)
            continue
        # boundary row: checked separately
        if K_g != K_o or sorted(idx_g) != sorted(int(x) for x in orc["indices"][n, :K_o]):
            differ.append(n)
        assert abs(K_g - K_o) <= 1, f"boundary row {n}: count {K_g} vs oracle {K_o}"
        b = int(orc["seq_of"][n])
        pos_of = {int(i): j for j, i in enumerate(mem.index[b])}
        sc = orc["scores"][n]
        top = [int(mem.index[b][j]) for j in S.order[:K_g]]
        cut = sc[S.order[K_g - 1]] if K_g else 0.0
        for x in set(idx_g) ^ set(top):
            assert abs(sc[pos_of[x]] - cut) < BAND * max(1.0, abs(cut)), \
                f"boundary row {n}: entry {x} outside the tie band"
        sel = np.array([pos_of[x] for x in idx_g], dtype=np.int64)
        r, _ = oracle.readout(sc, sel, mem.values[b])
        f = oracle.fuse(p, s.f64["h"][n:n + 1], r[None, :], mirror=mirror, rms_eps=RMS_EPS)
        ref_r[n], ref_h[n], ref_g[n] = r, f["h_out"][0], f["gate"][0]
    er = rel_err_rows(gpu["readout"][rows], ref_r[rows]) if gpu.get("readout") is not None else np.zeros(1)
    eh = rel_err_rows(gpu["h_out"][rows].astype(np.float64), ref_h[rows])
    eg = np.abs(gpu["gate"][rows] - ref_g[rows]).max() if len(rows) else 0.0
    assert er.max() <= tol, f"readout max rel err {er.max():.3e} > {tol} (row {rows[int(er.argmax())]})"
    assert eh.max() <= tol, f"h_out max rel err {eh.max():.3e} > {tol} (row {rows[int(eh.argmax())]})"
    assert eg <= GATE_TOL[w.dtype], f"gate max abs err {eg:.3e}"
    return dict(exempt=exempt, exempt_mass=n_mass, exempt_tie=n_tie, exempt_differ=differ,
                readout_err=float(er.max()), h_out_err=float(eh.max()),
                gate_err=float(eg), rows=len(rows))


def _check_order(orc, w, mem, n, idx_g):
    """GPU list is in descending score order up to tie-band swaps."""
    b = int(orc["seq_of"][n])
    pos_of = {int(i): j for j, i in enumerate(mem.index[b])}
    sc = orc["scores"][n]
    vals = [sc[pos_of[x]] for x in idx_g]
    for a, c in zip(vals, vals[1:]):
        assert a >= c - BAND * max(1.0, abs(a)) * 4, f"row {n}: selected list not in descending order"


def run_gpu(s: Stored, fovea, params=None, memory=None, l_max=None):
    """Build the memory and run one step through the C ABI; returns numpy outputs."""
    w = s.w
    params = params or params_for(s, fovea)
    mem = memory or fovea.build_memory(params, s.dev["v"], s.dev.get("mask"))
    out = fovea.step(params, mem, s.dev["h"], s.dev["depth"], w.row_offsets,
                     s.dev.get("row_scale"), w.rho, w.k_min, w.k_max, l_max=l_max)
    fovea.sync_errors(out["workspace"])
    res = {k: (v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy())
           for k, v in out.items() if v is not None and k != "workspace"}
    res["_memory"] = mem
    res["_params"] = params
    res["_folded"] = mem.folded_keys(params) is not None
    return res


def run_oracle(s: Stored, mirror: bool, rows=None, l_max=None):
    """The oracle in the paper's order of operations (q = W_Q x against the
    keys), in mirror mode for bf16 workloads."""
    w = s.w
    p = oracle_params(s)
    mem = oracle.build_memory(p, s.f64["v"], s.f64.get("mask"), mirror=mirror, ln_eps=LN_EPS)
    out = oracle.retrieve_fuse(p, mem, s.f64["h"], s.f64["depth"], w.row_offsets,
                               s.f64.get("row_scale"), w.rho, w.k_min, w.k_max, mirror=mirror,
                               rows=rows, ln_eps=LN_EPS, rms_eps=RMS_EPS, l_max=l_max)
    return out, mem
