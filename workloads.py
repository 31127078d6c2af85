"""Seeded synthetic workloads for the FOVEA retrieve+fuse path.

This module only draws inputs. It is shared by the CPU oracle's tests, the
CUDA parity tests and the benchmark, so it computes none of the path's
outputs: every array it returns is an *input* (weights, visual tokens,
masks, draft hidden states, depths, per-row temperatures).

The five recipes are shaped like the paper's VLM backbones (Sec. "Experimental
setup": LLaVA-NeXT-7B/13B and Qwen2.5-VL-7B drafters; candidate width 6,
tree depth D = 6) with all model widths equal, d_k = d_u = d_h = d_v = d
("Implementation and Training Details", visual correction module).  No
dataset and no trained weight is used: everything below is random.

Streams: workload k uses seed k - 1.  Each quantity draws from its own
PCG64 stream ``SeedSequence([seed, stream])``: 0 weights, 1 visual tokens,
2 hidden states, 3 depths (unused: depths are deterministic), 4 extras
(memory sizes, temperatures, planted entries), and 1000 + t for the hidden
states of draft step t of the long-memory workload.

Arrays come back as float32 (uint8 masks, int32 depths/offsets).  Callers
store them in the workload's dtype (bf16 or fp32); the stored values are the
inputs both the oracle and the CUDA path see.

Planted rows (LLaVA-7B-shaped workload).  A "peaked" draft state has one
memory entry whose key its query points at with cosine ~0.9.  Because W_Q
and W_K are random, aiming a query at a key needs the key and query maps
themselves (Sec. "Image-specific visual memory" and "State-conditioned
top-K visual evidence retrieval"), so the planting helper evaluates those two
maps in float64 *to construct the input*.  Nothing downstream reuses it: the
oracle and the kernels recompute every quantity from the stored inputs.
"""

from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np

MLP_HIDDEN = 512     # correction / gate hidden width ("Visual correction module")
MAX_DEPTH = 6        # tree depth D = 6 ("Experimental setup") -> E_dep has 7 rows
LN_EPS = 1e-5
RMS_EPS = 1e-6

STREAM_WEIGHTS, STREAM_VISUAL, STREAM_HIDDEN, STREAM_DEPTH, STREAM_EXTRA = 0, 1, 2, 3, 4

PARAM_NAMES = (
    "ln_v_gamma", "ln_v_beta", "W_K", "W_U",
    "ln_h_gamma", "ln_h_beta", "E_dep", "W_Q",
    "W_f1", "b_f1", "W_f2", "b_f2",
    "W_g1", "b_g1", "w_g2", "b_g2",
    "rms_gamma",
)


@dataclasses.dataclass(frozen=True)
class Spec:
    """One workload recipe (sizes, selection arguments, dtype, seed)."""
    index: int
    name: str
    d: int
    B: int
    rows_per_seq: int
    rho: float
    k_max: int
    k_min: int
    dtype: str                      # "bf16" or "fp32"
    seed: int
    m_fixed: Optional[int] = None   # memory entries per image when fixed
    m_choices: Optional[tuple] = None   # drawn per image from these sizes
    peaked_rows: int = 0            # rows per sequence with a planted entry
    planted_cos: float = 0.9
    log_temperature: Optional[tuple] = None   # (lo, hi) of ln T per row
    clusters: int = 0               # key clusters (long-memory workload)
    cluster_sigma: float = 0.0
    steps: int = 1                  # draft steps over one memory

    @property
    def N(self) -> int:
        return self.B * self.rows_per_seq

    @property
    def M_max(self) -> int:
        return self.m_fixed if self.m_fixed is not None else max(self.m_choices)


WORKLOADS: Dict[int, Spec] = {
    1: Spec(1, "tiny-fp32", d=256, B=1, rows_per_seq=4, rho=0.9, k_max=16,
            k_min=1, dtype="fp32", seed=0, m_fixed=64),
    2: Spec(2, "llava-1.5-7b-shaped", d=4096, B=1, rows_per_seq=64, rho=0.9,
            k_max=64, k_min=1, dtype="bf16", seed=1, m_fixed=576,
            peaked_rows=8),
    3: Spec(3, "qwen2-vl-7b-shaped", d=3584, B=8, rows_per_seq=32, rho=0.8,
            k_max=128, k_min=1, dtype="bf16", seed=2,
            m_choices=(256, 1024, 2880),
            log_temperature=(math.log(0.1), math.log(10.0))),
    4: Spec(4, "llava-1.5-13b-shaped", d=5120, B=16, rows_per_seq=64,
            rho=0.95, k_max=64, k_min=1, dtype="bf16", seed=3, m_fixed=576),
    5: Spec(5, "long-memory", d=4096, B=4, rows_per_seq=128, rho=0.9,
            k_max=256, k_min=1, dtype="bf16", seed=4, m_fixed=8192,
            clusters=64, cluster_sigma=0.2, steps=100),
}


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream])))


def draw_params(d: int, seed: int, H: int = MLP_HIDDEN, D: int = MAX_DEPTH) -> Dict[str, np.ndarray]:
    """Random weights: every linear W ~ N(0, 1/fan_in), biases ~ N(0, 0.01^2),
    LN gamma = 1 + 0.1 N(0,1), beta = 0.1 N(0,1), RMSNorm gamma = 1 + 0.1 N(0,1),
    E_dep ~ N(0, 0.1^2), and b_g2 = 0 so the gate starts near 1/2."""
    g = _rng(seed, STREAM_WEIGHTS)
    f32 = np.float32

    def lin(out_f, in_f):
        w = g.standard_normal((out_f, in_f), dtype=f32)
        w *= f32(1.0 / math.sqrt(in_f))
        return w

    p = {}
    p["ln_v_gamma"] = (1.0 + 0.1 * g.standard_normal(d)).astype(f32)
    p["ln_v_beta"] = (0.1 * g.standard_normal(d)).astype(f32)
    p["W_K"] = lin(d, d)
    p["W_U"] = lin(d, d)
    p["ln_h_gamma"] = (1.0 + 0.1 * g.standard_normal(d)).astype(f32)
    p["ln_h_beta"] = (0.1 * g.standard_normal(d)).astype(f32)
    p["E_dep"] = (0.1 * g.standard_normal((D + 1, d))).astype(f32)
    p["W_Q"] = lin(d, d)
    p["W_f1"] = lin(H, 2 * d)
    p["b_f1"] = (0.01 * g.standard_normal(H)).astype(f32)
    p["W_f2"] = lin(d, H)
    p["b_f2"] = (0.01 * g.standard_normal(d)).astype(f32)
    p["W_g1"] = lin(H, 2 * d)
    p["b_g1"] = (0.01 * g.standard_normal(H)).astype(f32)
    p["w_g2"] = (g.standard_normal(H) / math.sqrt(H)).astype(f32)
    p["b_g2"] = np.zeros(1, dtype=f32)
    p["rms_gamma"] = (1.0 + 0.1 * g.standard_normal(d)).astype(f32)
    return p


def tree_depths(rows: int) -> np.ndarray:
    """EAGLE-style tree order within one sequence: the root has depth 0, the
    next six rows (candidate width K_c = 6) depth 1, and the remaining rows
    cycle through depths 2..6 (D = 6)."""
    dep = np.empty(rows, dtype=np.int32)
    for j in range(rows):
        if j == 0:
            dep[j] = 0
        elif j <= 6:
            dep[j] = 1
        else:
            dep[j] = 2 + (j - 7) % (MAX_DEPTH - 1)
    return dep


@dataclasses.dataclass
class Workload:
    """Inputs of one workload (numpy, float32 unless stated)."""
    spec: Optional[Spec]
    name: str
    d: int
    dtype: str
    params: Dict[str, np.ndarray]
    v: np.ndarray               # [B, M_max, d]
    mask: Optional[np.ndarray]  # [B, M_max] uint8, or None = every entry valid
    m_sizes: List[int]          # valid entries per image
    h: np.ndarray               # [N, d]
    depth: np.ndarray           # [N] int32
    row_offsets: np.ndarray     # [B + 1] int32
    row_scale: Optional[np.ndarray]   # [N] float32 or None
    rho: float
    k_min: int
    k_max: int
    planted: Dict[int, int] = dataclasses.field(default_factory=dict)   # row -> entry

    @property
    def B(self) -> int:
        return self.v.shape[0]

    @property
    def M_max(self) -> int:
        return self.v.shape[1]

    @property
    def N(self) -> int:
        return self.h.shape[0]


# ----------------------------------------------------------------------------
# Planting (input construction only; see the module docstring)
# ----------------------------------------------------------------------------

def _ln64(x, gamma, beta, eps=LN_EPS):
    mu = x.mean(-1, keepdims=True)
    var = ((x - mu) ** 2).mean(-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * gamma + beta


def _plant_rows(p, v_entries, depths, noise, target_cos, mu=0.03):
    """Hidden states whose query points at the given entries' keys with the
    requested cosine.  ``v_entries`` [P, d] are the planted visual tokens,
    ``noise`` [P, d] isotropic draws.  Returns (h [P, d], achieved cos [P]).

    The LN output of a standardised h is gamma*h + beta, so the query is
    A h + b with A = W_Q diag(gamma_h) and b = W_Q (beta_h + E_dep[l]).  The
    direction z = (A^T A + mu I)^{-1} A^T t (conjugate gradients; mu trades
    alignment against the norm that LN removes) is standardised and then
    blended with orthogonal noise until cos(q, k) reaches the target."""
    W_Q = p["W_Q"].astype(np.float64)
    W_K = p["W_K"].astype(np.float64)
    E = p["E_dep"].astype(np.float64)
    gh, bh = p["ln_h_gamma"].astype(np.float64), p["ln_h_beta"].astype(np.float64)
    keys = _ln64(v_entries.astype(np.float64), p["ln_v_gamma"].astype(np.float64),
                 p["ln_v_beta"].astype(np.float64)) @ W_K.T
    t = keys / np.linalg.norm(keys, axis=1, keepdims=True)
    A = W_Q * gh[None, :]
    rhs = t @ A
    z = np.zeros_like(rhs)
    res = rhs.copy()
    direc = res.copy()
    rs = (res * res).sum(1)
    stop = 1e-20 * (rhs * rhs).sum(1)
    for _ in range(400):
        Ad = (direc @ A.T) @ A + mu * direc
        step = rs / (direc * Ad).sum(1)
        z += step[:, None] * direc
        res -= step[:, None] * Ad
        rn = (res * res).sum(1)
        if np.all(rn < stop):
            break
        direc = res + (rn / rs)[:, None] * direc
        rs = rn

    def standardise(x):
        x = x - x.mean(1, keepdims=True)
        return x / np.sqrt((x * x).mean(1, keepdims=True))

    u = standardise(z)
    xi = noise.astype(np.float64)
    xi = xi - xi.mean(1, keepdims=True)
    xi = standardise(xi - (xi * u).sum(1, keepdims=True) / (u * u).sum(1, keepdims=True) * u)

    def cos_at(beta):
        hh = beta[:, None] * u + np.sqrt(1.0 - beta[:, None] ** 2) * xi
        q = (_ln64(hh, gh, bh) + E[depths]) @ W_Q.T
        return (q * t).sum(1) / np.linalg.norm(q, axis=1), hh

    lo = np.zeros(len(depths))
    hi = np.ones(len(depths))
    for _ in range(40):
        mid = 0.5 * (lo + hi)
        c, _ = cos_at(mid)
        below = c < target_cos
        lo = np.where(below, mid, lo)
        hi = np.where(below, hi, mid)
    c, hh = cos_at(hi)
    return hh.astype(np.float32), c


# ----------------------------------------------------------------------------
# Generators
# ----------------------------------------------------------------------------

def _visual_tokens(spec_seed, B, M_max, d, clusters=0, sigma=0.0):
    g = _rng(spec_seed, STREAM_VISUAL)
    if clusters:
        centres = g.standard_normal((clusters, d), dtype=np.float32)
        z = g.integers(0, clusters, size=(B, M_max))
        v = centres[z] + np.float32(sigma) * g.standard_normal((B, M_max, d), dtype=np.float32)
        return v.astype(np.float32)
    return g.standard_normal((B, M_max, d), dtype=np.float32)


def hidden_states(seed: int, N: int, d: int, step: Optional[int] = None) -> np.ndarray:
    """Isotropic draft hidden states h ~ N(0, 1); draft step ``step`` of a
    multi-step workload uses stream 1000 + step."""
    stream = STREAM_HIDDEN if step is None else 1000 + step
    return _rng(seed, stream).standard_normal((N, d), dtype=np.float32)


def generate(spec: Spec, step: Optional[int] = None, params=None, v=None) -> Workload:
    """Inputs of a named workload.  ``params``/``v`` may be passed in to reuse
    a previous draw (the long-memory workload keeps one memory over steps)."""
    d, B = spec.d, spec.B
    ex = _rng(spec.seed, STREAM_EXTRA)
    if spec.m_fixed is not None:
        m_sizes = [spec.m_fixed] * B
    else:
        m_sizes = [int(x) for x in ex.choice(np.array(spec.m_choices), size=B)]
    M_max = spec.M_max
    if params is None:
        params = draw_params(d, spec.seed)
    if v is None:
        v = _visual_tokens(spec.seed, B, M_max, d, spec.clusters, spec.cluster_sigma)
    mask = None
    if any(m != M_max for m in m_sizes):
        mask = np.zeros((B, M_max), dtype=np.uint8)
        for b, m in enumerate(m_sizes):
            mask[b, :m] = 1          # trailing padding
    R = spec.rows_per_seq
    N = B * R
    h = hidden_states(spec.seed, N, d, step if spec.steps > 1 else None)
    depth = np.concatenate([tree_depths(R) for _ in range(B)]).astype(np.int32)
    row_offsets = (np.arange(B + 1) * R).astype(np.int32)
    row_scale = None
    if spec.log_temperature is not None:
        lo, hi = spec.log_temperature
        T = np.exp(ex.uniform(lo, hi, size=N))
        row_scale = (1.0 / T).astype(np.float32)
    planted = {}
    if spec.peaked_rows:
        rows, entries = [], []
        for b in range(B):
            picks = ex.choice(m_sizes[b], size=spec.peaked_rows, replace=False)
            for j in range(spec.peaked_rows):
                rows.append(b * R + j)
                entries.append((b, int(picks[j])))
        noise = h[rows]
        vv = np.stack([v[b, e] for b, e in entries])
        hp, _ = _plant_rows(params, vv, depth[rows], noise, spec.planted_cos)
        h = h.copy()
        h[rows] = hp
        planted = {r: e for r, (_, e) in zip(rows, entries)}
    return Workload(spec, spec.name, d, spec.dtype, params, v, mask, m_sizes, h,
                    depth, row_offsets, row_scale, spec.rho, spec.k_min,
                    spec.k_max, planted)


def generate_custom(name: str, d: int, m_sizes: List[int], rows: List[int], *,
                    M_max: Optional[int] = None, rho: float = 0.9,
                    k_max: int = 16, k_min: int = 1, dtype: str = "bf16",
                    seed: int = 7, temperature: Optional[tuple] = None,
                    clusters: int = 0, cluster_sigma: float = 0.0,
                    scattered_mask: bool = False, H: int = MLP_HIDDEN) -> Workload:
    """A small workload with explicit per-image memory sizes and per-sequence
    draft rows (ragged allowed), for parity tests that must span several
    tiles and ragged tails.  ``scattered_mask`` spreads the valid entries of
    each image over random positions instead of trailing padding."""
    B = len(m_sizes)
    assert len(rows) == B
    if M_max is None:
        M_max = max(max(m_sizes), 1)
    params = draw_params(d, seed, H=H)
    v = _visual_tokens(seed, B, M_max, d, clusters, cluster_sigma)
    ex = _rng(seed, STREAM_EXTRA)
    mask = None
    if scattered_mask or any(m != M_max for m in m_sizes):
        mask = np.zeros((B, M_max), dtype=np.uint8)
        for b, m in enumerate(m_sizes):
            if scattered_mask:
                mask[b, ex.choice(M_max, size=m, replace=False)] = 1
            else:
                mask[b, :m] = 1
    N = int(sum(rows))
    h = hidden_states(seed, N, d)
    depth = np.concatenate([tree_depths(r) for r in rows] or [np.zeros(0, np.int32)]).astype(np.int32)
    row_offsets = np.concatenate([[0], np.cumsum(rows)]).astype(np.int32)
    row_scale = None
    if temperature is not None:
        lo, hi = temperature
        T = np.exp(ex.uniform(math.log(lo), math.log(hi), size=N))
        row_scale = (1.0 / T).astype(np.float32)
    return Workload(None, name, d, dtype, params, v, mask, list(m_sizes), h, depth,
                    row_offsets, row_scale, rho, k_min, k_max, {})
