"""Oracle of the data-free importance and the outlier-column selection.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  The product path
(the CUDA library and its binding) never does; the two share no code.

Plain numpy in float64, written from the paper's definitions:

* Eq. gamma (Sec. 3.2, input side): a_j = gamma_j^2 for the five projections
  that read gamma * RMSNorm(h) (q, k, v, gate, up); the language-model head
  reads the final norm's output the same way.
* Eq. prop (Sec. 3.2): a^(o) = repeat_kv((W_v o W_v) a^(in)) and
  a^(down)_c = E[silu(g_c)^2] ((W_up o W_up) a^(in))_c with
  g_c ~ N(0, ((W_gate o W_gate) a^(in))_c), the expectation by Gauss-Hermite
  quadrature.
* Output side (Sec. 3.2 and App. A.1): an isotropic gradient at the logits, one
  hop through the head, then every layer in reverse order maps the residual
  gradient scale back through its own matrices with
  E[g_in,c^2] = sum_r W_rc^2 E[g_out,r^2]; the rows of W_o and W_down take the
  residual scale they write to as rho; all other rows have rho = 1 (the
  conservative variant of App. A.1).
* The stored rho is normalized to unit mean within its tensor (reading: the
  paper normalizes both factors to unit mean before use, and the raw proxy
  leaves float32 range on deep models).
* Outlier columns (Sec. 3.5, App. A.6): the dynamic-range rule
  max_i |W_ij| / (median_i |W_ij| + eps) >= 1e3 and the activation rule
  a_j >= 1e2 times the tensor mean; at most 32 per rule, ranked by the better
  position in the two lists, the first four kept for the whole model.

The factors are stored in single precision (App. A.7), so every table this
module returns is float32 rounded from the float64 result.

Readings where the paper leaves a choice open (each also listed in the design
notes): the quadrature uses ``GH_NODES`` nodes; the normalisations are the
identity in the backward proxy (their Jacobians are dropped, gains included);
the residual connection adds the branch's gradient scale to the stream's; the
attention back-map sums the query heads that share a key-value head; the median
of an even count is the mean of the two middle values; eps is the smallest
positive FP16 number; the activation statistic is a_j divided by the tensor
mean, the mean the correctly rounded sum over the columns divided by their
count; ties in the merged ranking fall to the
tensor index, then the column index.
"""
from __future__ import annotations

import numpy as np

GH_NODES = 64          # Gauss-Hermite nodes for E[silu(g)^2] (reading)
EPS_DR = 2.0 ** -24    # eps of the dynamic-range rule (reading: smallest FP16 step)
DR_MIN = 1.0e3         # Sec. 3.5 dynamic-range threshold
ACT_MIN = 1.0e2        # Sec. 3.5 activation threshold (times the tensor mean)
LIST_MAX = 32          # App. A.6: each rule keeps at most its 32 largest values
N_OUTLIERS = 4         # App. A.6: the first four candidates are stored

# Tensor order of one layer; the model's tensors are these per layer, then the head.
KINDS = ("q", "k", "v", "o", "gate", "up", "down")


def f16(bits) -> np.ndarray:
    """FP16 bit patterns (uint16) as float64 values."""
    return np.asarray(bits, np.uint16).view(np.float16).astype(np.float64)


# --------------------------------------------------------------- Eq. gamma / prop

def a_from_gain(gamma_bits) -> np.ndarray:
    """Eq. gamma: a_j = gamma_j^2 (the normalised channels taken as unit second moment)."""
    g = f16(gamma_bits)
    return g * g


def sq_rows(W_bits, v) -> np.ndarray:
    """(W o W) v: second moment of each output of y = W x for independent x_c
    with E[x_c^2] = v_c (the one-hop propagation of Eq. prop)."""
    W = f16(W_bits)
    return (W * W) @ np.asarray(v, np.float64)


def sq_cols(W_bits, g) -> np.ndarray:
    """(W o W)^T g: second moment of each input gradient of y = W x for
    independent output gradients with E[g_r^2] = g_r (the backward proxy)."""
    W = f16(W_bits)
    return (W * W).T @ np.asarray(g, np.float64)


def silu_sq_moment(var) -> np.ndarray:
    """E[silu(g)^2] for g ~ N(0, var) by Gauss-Hermite quadrature (Eq. prop):
    int f(x) exp(-x^2) dx ~ sum_i w_i f(x_i) with g = sqrt(2 var) x."""
    t, w = np.polynomial.hermite.hermgauss(GH_NODES)
    var = np.asarray(var, np.float64)
    g = np.sqrt(2.0 * var)[..., None] * t
    s = g / (1.0 + np.exp(-g))
    return (s * s) @ w / np.sqrt(np.pi)


def repeat_kv(v_kv, n_heads: int, n_kv_heads: int) -> np.ndarray:
    """Channels of the key-value heads repeated for the query heads that read
    them: query head h reads key-value head h // (n_heads / n_kv_heads)."""
    hd = v_kv.size // n_kv_heads
    return np.repeat(np.asarray(v_kv).reshape(n_kv_heads, hd), n_heads // n_kv_heads, axis=0).ravel()


def a_o(Wv_bits, a_in, n_heads: int, n_kv_heads: int) -> np.ndarray:
    """Eq. prop, attention output projection: repeat_kv((W_v o W_v) a^(in))."""
    return repeat_kv(sq_rows(Wv_bits, a_in), n_heads, n_kv_heads)


def a_down(Wgate_bits, Wup_bits, a_in) -> np.ndarray:
    """Eq. prop, MLP down projection: E[silu(g_c)^2] ((W_up o W_up) a^(in))_c,
    g_c ~ N(0, ((W_gate o W_gate) a^(in))_c)."""
    return silu_sq_moment(sq_rows(Wgate_bits, a_in)) * sq_rows(Wup_bits, a_in)


def rho_proxy(model) -> list:
    """Output-side factor of Sec. 3.2 / App. A.1: per layer (rho_o, rho_down),
    each a d_model vector, from the backward second-moment proxy."""
    s = model.spec
    G = sq_cols(model.lm_head(), np.ones(s.vocab))
    out = [None] * s.n_layers
    n_rep = s.n_heads // s.n_kv_heads
    for l in reversed(range(s.n_layers)):
        rho_down = G.copy()
        Gh = sq_cols(model.weight(l, "down"), G)
        G = G + sq_cols(model.weight(l, "gate"), Gh) + sq_cols(model.weight(l, "up"), Gh)
        rho_o = G.copy()
        Ga = sq_cols(model.weight(l, "o"), G)
        Gv = Ga.reshape(s.n_kv_heads, n_rep, s.head_dim).sum(axis=1).ravel()
        G = G + sq_cols(model.weight(l, "v"), Gv)
        out[l] = (rho_o, rho_down)
    return out


def unit_mean(v) -> np.ndarray:
    """v divided by its mean, the mean summed in index order (the stored rho:
    only its shape within the tensor matters, Eq. imp and App. A.2)."""
    v = np.asarray(v, np.float64)
    return v / (np.cumsum(v)[-1] / v.size)


def importance_tables(model) -> list:
    """(name, a, rho) for every tensor of the model in its tensor order (per
    layer q, k, v, o, gate, up, down; then the head), a and rho in float32 as
    stored (rho None where it is 1 on every row; otherwise normalized to unit
    mean, which keeps the table in float32 range: the proxy's scale grows by a
    model-dependent factor per layer)."""
    s = model.spec
    rho = [(unit_mean(ro), unit_mean(rd)) for ro, rd in rho_proxy(model)]
    out = []
    for l in range(s.n_layers):
        a_attn = a_from_gain(model.gain(l, "attn"))
        a_mlp = a_from_gain(model.gain(l, "mlp"))
        ao = a_o(model.weight(l, "v"), a_attn, s.n_heads, s.n_kv_heads)
        ad = a_down(model.weight(l, "gate"), model.weight(l, "up"), a_mlp)
        f32 = lambda v: np.asarray(v, np.float64).astype(np.float32)
        out += [(f"l{l}.q", f32(a_attn), None), (f"l{l}.k", f32(a_attn), None),
                (f"l{l}.v", f32(a_attn), None), (f"l{l}.o", f32(ao), f32(rho[l][0])),
                (f"l{l}.gate", f32(a_mlp), None), (f"l{l}.up", f32(a_mlp), None),
                (f"l{l}.down", f32(ad), f32(rho[l][1]))]
    out.append(("lm_head", a_from_gain(model.gain(None, "final")).astype(np.float32), None))
    return out


# ------------------------------------------------------------- outlier columns

def column_max_median(W_bits):
    """Per column j: max_i |W_ij| and median_i |W_ij| (mean of the two middle
    values when the row count is even), from a full sort."""
    A = np.abs(f16(W_bits))
    S = np.sort(A, axis=0)
    R = S.shape[0]
    med = 0.5 * (S[(R - 1) // 2] + S[R // 2])
    return S[-1], med


def dynamic_range(W_bits) -> np.ndarray:
    """Sec. 3.5 statistic of every column: max / (median + eps)."""
    mx, med = column_max_median(W_bits)
    return mx / (med + EPS_DR)


def activation_ratio(a) -> np.ndarray:
    """a_j divided by the tensor mean of a; the mean is the correctly rounded
    sum of a (math.fsum) divided by the column count."""
    import math

    a64 = np.asarray(a, np.float32).astype(np.float64)
    mean = math.fsum(a64.tolist()) / a64.size
    return a64 / mean


def rule_list(stats) -> list:
    """One rule's list: [(value, tensor, column)] over all tensors, largest
    first, ties by tensor then column, at most LIST_MAX.  ``stats`` is a list
    of (per-column statistic, threshold) per tensor."""
    cand = []
    for t, (v, thr) in enumerate(stats):
        for c in np.nonzero(v >= thr)[0]:
            cand.append((-float(v[c]), t, int(c)))
    cand.sort()
    return [(-x, t, c) for x, t, c in cand[:LIST_MAX]]


def select_outliers(dr_per_tensor, ratio_per_tensor, n_keep: int = N_OUTLIERS) -> list:
    """App. A.6: both lists, each candidate ranked by its better position in
    them, ties by tensor then column; the first n_keep (tensor, column)."""
    L1 = rule_list([(d, DR_MIN) for d in dr_per_tensor])
    L2 = rule_list([(r, ACT_MIN) for r in ratio_per_tensor])
    best = {}
    for lst in (L1, L2):
        for pos, (_, t, c) in enumerate(lst):
            best[(t, c)] = min(best.get((t, c), pos), pos)
    ranked = sorted(best, key=lambda tc: (best[tc], tc[0], tc[1]))
    return ranked[:n_keep]


def model_outliers(model, tables=None) -> list:
    """The model's stored outlier columns: (tensor index, column) pairs."""
    if tables is None:
        tables = importance_tables(model)
    ws = [model.tensor(i) for i in range(len(tables))]
    return select_outliers([dynamic_range(W) for W in ws], [activation_ratio(a) for _, a, _ in tables])
