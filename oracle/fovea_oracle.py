"""Plain float64 CPU oracle of the FOVEA retrieve+fuse path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product (the C-ABI library and its
Python binding) imports, calls or links this module; only ``tests/``, the
``smoke()`` check of ``__graft_entry__`` and the CPU-baseline leg of
``bench.py`` may use it.  It shares no code with the CUDA path.

Every function follows the paper's definitions in the paper's order and
notation, with numpy float64 arithmetic and numpy's matrix product as the
only library primitive.  Nothing is blocked, fused or reordered.

* Memory: k_i = W_K LN(v_i), u_i = W_U LN(v_i) over valid i (Eq. of the
  image-specific visual memory, Sec. "Image-specific visual memory").
* Query and scores: q_n = W_Q(LN(h_n) + E_dep[l_n]), s_{n,i} = q_n k_i / sqrt(d_k)
  (Sec. "State-conditioned top-K visual evidence retrieval", first equation).
* Global softmax over the valid set, descending order pi_n, cumulative-mass
  cardinality K_raw and its clamp K (the alpha-tilde and K_{r,n} equations).
* Renormalised weights over the selected set and readout r_n (the alpha and
  r_n equation).
* Correction c_n = f([h; r]), gate g_n = sigma(g([h; r])), and
  h_hat = RMSNorm(h + g c) (Eq. hidden_correction; the appendix's
  "Visual correction module" fixes two biased linears, a 512 hidden layer,
  SiLU, a d-dim correction and a scalar gate broadcast over d).

Readings where the paper leaves a detail open (each also listed in the
design notes):

* score scale 1/sqrt(d_k) with d_k = d; ``row_scale`` multiplies it (1 when
  absent) - an extension used for per-row temperatures;
* pi_n orders by descending score s, ties by smaller original index;
* K_raw is the first k in 1..|V| with C_k >= rho, |V| when rounding keeps C
  below rho; an empty valid set gives K = 0 and r = 0;
* LN has affine gamma/beta (eps 1e-5); LN of visual tokens and LN of hidden
  states are separate parameter sets; RMSNorm has a weight (eps 1e-6);
* f and g read the same [h; r] (h first) with separate first layers.

``mirror=True`` rounds to bfloat16 (round to nearest, ties to even) at the
points where the bf16 storage path stores a value: LN(v) (R1), k and u (R2),
LN(h) + E_dep (R3), r before the fusion (R6), the SiLU activations (R7) and
h_hat (R8).  The query q is not rounded: the bf16 path carries it as a pair
of bf16 values (about 16 significant bits), so its scores follow the exact
q.  ``mirror=False`` is exact float64 throughout.

Query folding (``fold=True`` in ``retrieve_fuse``): since q_n . k_i =
(W_Q x_n) . k_i = x_n . (W_Q^T k_i) with x_n = LN(h_n) + E_dep[l_n], the scores
may be taken against folded keys kappa_i = W_Q^T k_i formed once per image
(``fold_keys``).  In exact arithmetic both orders give the same scores; in
mirror mode kappa_i is rounded to bfloat16 (R9, the folded keys' storage)
and x_n keeps its R3 rounding, which is what the folded bf16 path stores.

Depth gate (``l_max`` in ``retrieve_fuse``; the experimental setup applies
the visual correction only to nodes of depth at most 1): a draft state whose
depth exceeds l_max is not corrected, so its scoring representation is h_n
itself, with no retrieval (count 0, no indices, r = 0, gate 0).

The draft logits z_n = W_LM h_hat_n and their K_c largest entries
(``lm_head_topk``) follow Eq. hidden_correction and the candidate width of
the experimental setup; the order is by logit, ties by smaller token index.

Parity pins: tests/test_oracle_pins.py (bf16 rounding against torch, LN/RMSNorm
against torch.nn.functional, subset enumeration, closed forms, dense
attention, fixed top-K against lexsort, gate identities).
"""

from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np

F64 = np.float64
BF16_MAX = float.fromhex("0x1.fe00000000000p+127")


# ----------------------------------------------------------------------------
# Storage rounding
# ----------------------------------------------------------------------------

def round_bf16(x) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 value (8 significant
    bits, 8 exponent bits, ties to even), returned as float64."""
    x = np.asarray(x, dtype=F64)
    out = x.copy()
    fin = np.isfinite(x) & (x != 0.0)
    xs = x[fin]
    _, e = np.frexp(xs)                      # |x| = m 2^e, 0.5 <= m < 1
    spacing_exp = np.maximum(e, -125) - 8    # normals: 2^(e-8); subnormals: 2^-133
    r = np.ldexp(np.rint(np.ldexp(xs, -spacing_exp)), spacing_exp)
    r = np.where(np.abs(r) > BF16_MAX, np.copysign(np.inf, r), r)
    out[fin] = r
    return out


# ----------------------------------------------------------------------------
# Elementary operators
# ----------------------------------------------------------------------------

def layer_norm(x, gamma, beta, eps):
    """LN over the last axis: (x - mean) / sqrt(var + eps) * gamma + beta,
    var the biased (population) variance."""
    x = np.asarray(x, dtype=F64)
    mean = x.mean(axis=-1, keepdims=True)
    var = ((x - mean) ** 2).mean(axis=-1, keepdims=True)
    return (x - mean) / np.sqrt(var + eps) * gamma + beta


def rms_norm(y, gamma, eps):
    """RMSNorm over the last axis: y / sqrt(mean(y^2) + eps) * gamma."""
    y = np.asarray(y, dtype=F64)
    return y / np.sqrt((y ** 2).mean(axis=-1, keepdims=True) + eps) * gamma


def sigmoid(x):
    x = np.asarray(x, dtype=F64)
    out = np.empty_like(x)
    pos = x >= 0
    out[pos] = 1.0 / (1.0 + np.exp(-x[pos]))
    ex = np.exp(x[~pos])
    out[~pos] = ex / (1.0 + ex)
    return out


def silu(x):
    x = np.asarray(x, dtype=F64)
    return x * sigmoid(x)


def _maybe(x, mirror):
    return round_bf16(x) if mirror else x


# ----------------------------------------------------------------------------
# Visual memory (Sec. "Image-specific visual memory")
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class Memory:
    keys: List[np.ndarray]      # per image [|V_b|, d], k_i
    values: List[np.ndarray]    # per image [|V_b|, d], u_i
    index: List[np.ndarray]     # per image: original position i of each valid entry
    d: int
    folded: Optional[List[np.ndarray]] = None   # per image [|V_b|, d], kappa_i = W_Q^T k_i


def build_memory(p: Dict[str, np.ndarray], v, mask=None, *, mirror=False,
                 ln_eps=1e-5) -> Memory:
    """M_img = {(k_i, u_i, m_i)}: k_i = W_K LN(v_i), u_i = W_U LN(v_i), kept
    for the valid positions V = {i | m_i = 1} in ascending i."""
    v = np.asarray(v, dtype=F64)
    B, M_max, d = v.shape
    keys, values, index = [], [], []
    for b in range(B):
        valid = np.arange(M_max) if mask is None else np.flatnonzero(np.asarray(mask[b]) != 0)
        x = _maybe(layer_norm(v[b, valid], p["ln_v_gamma"], p["ln_v_beta"], ln_eps), mirror)
        k = _maybe(x @ p["W_K"].T, mirror)
        u = _maybe(x @ p["W_U"].T, mirror)
        keys.append(k)
        values.append(u)
        index.append(valid.astype(np.int64))
    return Memory(keys, values, index, d)


# ----------------------------------------------------------------------------
# Retrieval (Sec. "State-conditioned top-K visual evidence retrieval")
# ----------------------------------------------------------------------------

def query_input(p, h, depth, *, mirror=False, ln_eps=1e-5):
    """x_n = LN(h_n) + E_dep[l_n], the input of the query projection."""
    return _maybe(layer_norm(h, p["ln_h_gamma"], p["ln_h_beta"], ln_eps)
                  + p["E_dep"][np.asarray(depth)], mirror)


def query(p, h, depth, *, mirror=False, ln_eps=1e-5):
    """q_n = W_Q (LN(h_n) + E_dep[l_n])."""
    return query_input(p, h, depth, mirror=mirror, ln_eps=ln_eps) @ p["W_Q"].T


def fold_keys(p, mem: Memory, *, mirror=False, images=None) -> Memory:
    """Query folding: kappa_i = W_Q^T k_i for every key of the given images
    (default all), so that q_n . k_i = x_n . kappa_i.  Returns the memory with
    ``folded`` set (None for images not folded)."""
    B = len(mem.keys)
    images = range(B) if images is None else set(images)
    folded = [_maybe(mem.keys[b] @ p["W_Q"], mirror) if b in images else None for b in range(B)]
    return dataclasses.replace(mem, folded=folded)


def scores(q_n, K_b, d, row_scale_n=1.0):
    """s_{n,i} = q_n k_i / sqrt(d_k) (times the optional per-row scale)."""
    return (K_b @ q_n) / math.sqrt(d) * row_scale_n


@dataclasses.dataclass
class Selection:
    K: int                  # K_{r,n}
    K_raw: int              # K^raw_{r,n}
    order: np.ndarray       # pi_n over positions 0..|V|-1 (descending s, ascending index)
    cum_mass: np.ndarray    # C_k = sum_{t<=k} alpha-tilde_{pi(t)}, k = 1..|V|
    alpha_tilde: np.ndarray # global softmax over V, in position order
    selected: np.ndarray    # I_n = pi_n(1..K), positions


def select(s, rho, k_min, k_max) -> Selection:
    """alpha-tilde = softmax over V; pi = descending order; K_raw = min{k :
    sum_{t<=k} alpha-tilde_{pi(t)} >= rho}; K = min(|V|, K_max, max(K_min, K_raw))."""
    s = np.asarray(s, dtype=F64)
    V = s.shape[0]
    if V == 0:
        e = np.zeros(0)
        return Selection(0, 0, np.zeros(0, np.int64), e, e, np.zeros(0, np.int64))
    ex = np.exp(s - s.max())
    alpha_tilde = ex / ex.sum()
    order = np.lexsort((np.arange(V), -s))       # primary: -s ascending; then index
    cum = np.cumsum(alpha_tilde[order])
    hit = np.flatnonzero(cum >= rho)
    K_raw = int(hit[0]) + 1 if hit.size else V
    K = min(V, k_max, max(k_min, K_raw))
    return Selection(K, K_raw, order, cum, alpha_tilde, order[:K])


def readout(s, selected, U_b):
    """alpha_{n,i} = exp(s_i) / sum_{j in I} exp(s_j) over I; r_n = sum alpha_i u_i.
    Returns (r, alpha); an empty I gives r = 0."""
    d = U_b.shape[1] if U_b.ndim == 2 else 0
    if len(selected) == 0:
        return np.zeros(d), np.zeros(0)
    s_sel = np.asarray(s, dtype=F64)[selected]
    ex = np.exp(s_sel - s_sel.max())
    alpha = ex / ex.sum()
    return alpha @ U_b[selected], alpha


# ----------------------------------------------------------------------------
# Gated residual correction (Eq. hidden_correction)
# ----------------------------------------------------------------------------

def fuse(p, h, r, *, mirror=False, rms_eps=1e-6):
    """c = f([h; r]), g = sigma(g([h; r])), h_hat = RMSNorm(h + g c), with f and g
    each Linear(2d -> 512) + bias, SiLU, Linear(512 -> d or 1) + bias."""
    h = np.asarray(h, dtype=F64)
    z = np.concatenate([h, _maybe(r, mirror)], axis=-1)
    a_f = _maybe(silu(z @ p["W_f1"].T + p["b_f1"]), mirror)
    a_g = _maybe(silu(z @ p["W_g1"].T + p["b_g1"]), mirror)
    c = a_f @ p["W_f2"].T + p["b_f2"]
    g = sigmoid(a_g @ p["w_g2"] + p["b_g2"][0])
    y = h + g[:, None] * c
    h_hat = _maybe(rms_norm(y, p["rms_gamma"], rms_eps), mirror)
    return dict(a_f=a_f, a_g=a_g, c=c, gate=g, y=y, h_out=h_hat)


# ----------------------------------------------------------------------------
# One draft step over a batch of draft states
# ----------------------------------------------------------------------------

def retrieve_fuse(p, mem: Memory, h, depth, row_offsets, row_scale, rho, k_min,
                  k_max, *, mirror=False, ln_eps=1e-5, rms_eps=1e-6,
                  rows=None, fold=False, l_max=None) -> Dict[str, object]:
    """Retrieve + fuse for every draft state; rows row_offsets[b] ..
    row_offsets[b+1]-1 query image b.  ``rows`` restricts the computation to a
    subset of row indices (the rest of the outputs stay zero / -1).
    ``fold`` scores x_n against the folded keys (``fold_keys``) instead of
    q_n against the keys.  ``l_max``: rows deeper than l_max are not
    corrected (h_out = h, no retrieval); None corrects every row."""
    h = np.asarray(h, dtype=F64)
    N, d = h.shape
    rho = float(np.float32(rho))
    row_offsets = np.asarray(row_offsets)
    want = np.arange(N) if rows is None else np.asarray(sorted(rows))
    gated = np.zeros(N, bool)
    if l_max is not None:
        gated = np.asarray(depth) > l_max
    keep = want[~gated[want]] if len(want) else want
    seq_of = np.searchsorted(row_offsets, np.arange(N), side="right") - 1
    q = np.zeros((N, d))
    x = np.zeros((N, d))
    if fold and mem.folded is None:
        mem = fold_keys(p, mem, mirror=mirror, images={int(seq_of[n]) for n in keep})
    if len(keep):
        x[keep] = query_input(p, h[keep], np.asarray(depth)[keep], mirror=mirror, ln_eps=ln_eps)
        q[keep] = x[keep] @ p["W_Q"].T
    counts = np.zeros(N, np.int64)
    k_raw = np.zeros(N, np.int64)
    indices = -np.ones((N, k_max), np.int64)
    r = np.zeros((N, d))
    sel: List[Optional[Selection]] = [None] * N
    sc: List[Optional[np.ndarray]] = [None] * N
    alphas: List[Optional[np.ndarray]] = [None] * N
    for n in keep:
        b = int(seq_of[n])
        scale = 1.0 if row_scale is None else float(row_scale[n])
        s = scores(x[n], mem.folded[b], d, scale) if fold else scores(q[n], mem.keys[b], d, scale)
        S = select(s, rho, k_min, k_max)
        r[n], alphas[n] = readout(s, S.selected, mem.values[b])
        counts[n], k_raw[n] = S.K, S.K_raw
        indices[n, :S.K] = mem.index[b][S.selected]
        sel[n], sc[n] = S, s
    out = dict(q=q, counts=counts, k_raw=k_raw, indices=indices, readout=r,
               selections=sel, scores=sc, alphas=alphas, seq_of=seq_of, gated=gated)
    f = fuse(p, h[keep], r[keep], mirror=mirror, rms_eps=rms_eps)
    for key in ("a_f", "a_g", "c", "y", "h_out"):
        full = np.zeros((N,) + f[key].shape[1:])
        full[keep] = f[key]
        out[key] = full
    skipped = want[gated[want]] if len(want) else want
    out["h_out"][skipped] = h[skipped]          # not corrected: h_hat = h
    gate = np.zeros(N)
    gate[keep] = f["gate"]
    out["gate"] = gate
    return out


# ----------------------------------------------------------------------------
# Draft logits and tree-expansion candidates (Eq. hidden_correction: z = W_LM h_hat;
# the experimental setup's candidate width K_c)
# ----------------------------------------------------------------------------

def lm_head_topk(W_LM, h_hat, k_c) -> Dict[str, np.ndarray]:
    """z_n = W_LM h_hat_n over the vocabulary, and the K_c candidates of each
    row: the largest logits in descending order, ties broken by the smaller
    token index.  Returns logits [N, V], top_idx [N, K_c], top_val [N, K_c]."""
    W_LM = np.asarray(W_LM, dtype=F64)
    h_hat = np.asarray(h_hat, dtype=F64)
    z = h_hat @ W_LM.T
    V = W_LM.shape[0]
    k = min(int(k_c), V)
    top_idx = np.zeros((z.shape[0], k), np.int64)
    for n in range(z.shape[0]):
        order = np.lexsort((np.arange(V), -z[n]))    # primary: -z ascending; then index
        top_idx[n] = order[:k]
    top_val = np.take_along_axis(z, top_idx, axis=1)
    return dict(logits=z, top_idx=top_idx, top_val=top_val)

