"""Oracle: offline drift metrics on paired FP16 / low-bit logits, and the
recovery-window calibration rule.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Follows Sec. 4.1 ("Adaptive recovery-window selection") and Sec. 4.2
("Offline supervision and calibration") of the paper, all in float64.  For
one decode step t with FP16 logits z_fp and low-bit logits z_q:

1. p_fp = softmax(z_fp), p_q = softmax(z_q);
2. the FP16 candidate set C(alpha): the shortest prefix of the FP16 order
   (probability descending) whose cumulative mass reaches alpha; M_t is its
   size;
3. the active recovery region S = TopK(z_q, K);
4. recoverable coverage c_t = sum of p_fp over C intersect S;
5. local drift d_loc = || p_fp|U / p_fp(U) - p_q|U / p_q(U) ||_2 over
   U = C union S (each vector renormalised over U);
6. the label y_t = [d_loc > eps and c_t >= rho_c];
7. the coverage curve cov_t(K) = sum of p_fp over C intersect TopK(z_q, K)
   for K = 1 .. K_max, and the window K_b = the smallest K whose mean
   coverage over the steps reaches rho_K (0 when none does).

Readings taken where the paper is silent:

* both orders (the FP16 order and TopK) put equal values lowest index first,
  as the runtime TopK does;
* if the cumulative FP16 mass never reaches alpha (alpha = 1 and rounding),
  C is the whole vocabulary;
* alpha, eps, rho_c and rho_K are parameters: the paper prints no values.
"""

import numpy as np


def softmax(z):
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - z.max())
    return e / e.sum()


def order_desc(z):
    """Indices by value descending, lowest index first among equal values
    (a stable sort of -z)."""
    return np.argsort(-np.asarray(z, dtype=np.float64), kind="stable")


def candidate_set(p_fp, order_fp, alpha):
    """C(alpha) of Sec. 4.1: the first M_t indices of the FP16 order, M_t the
    least M whose prefix mass reaches alpha.  Returns (C, M_t)."""
    csum = np.cumsum(p_fp[order_fp])
    hit = np.nonzero(csum >= alpha)[0]
    m = int(hit[0]) + 1 if hit.size else len(order_fp)
    return order_fp[:m], m


def step_metrics(z_fp, z_q, alpha, K, eps, rho_c, k_max=None):
    """c_t, d_loc and y_t of Sec. 4.2 for one step, plus M_t and the coverage
    curve cov(K') for K' = 1 .. k_max (Sec. 4.1)."""
    z_fp = np.asarray(z_fp, dtype=np.float64)
    C, _ = candidate_set(softmax(z_fp), order_desc(z_fp), alpha)
    return metrics_given_candidates(z_fp, z_q, C, K, eps, rho_c, k_max)


def metrics_given_candidates(z_fp, z_q, C, K, eps, rho_c, k_max=None):
    """Steps 3-7 for a given FP16 candidate set C (Sec. 4.1-4.2): c_t, d_loc,
    y_t and the coverage curve with C fixed rather than found from alpha;
    M_t is |C|."""
    z_fp = np.asarray(z_fp, dtype=np.float64)
    z_q = np.asarray(z_q, dtype=np.float64)
    V = z_fp.shape[0]
    p_fp, p_q = softmax(z_fp), softmax(z_q)
    in_c = np.zeros(V, bool)
    in_c[C] = True
    order_q = order_desc(z_q)
    S = order_q[:K]
    in_s = np.zeros(V, bool)
    in_s[S] = True
    c = float(p_fp[in_c & in_s].sum())
    U = in_c | in_s
    a = p_fp[U] / p_fp[U].sum()
    b = p_q[U] / p_q[U].sum()
    d = float(np.sqrt(((a - b) ** 2).sum()))
    y = bool(d > eps and c >= rho_c)
    out = {"M": len(C), "c": c, "d_loc": d, "y": y, "C": C, "S": S}
    if k_max is not None:
        top = order_q[:k_max]
        out["cov"] = np.cumsum(np.where(in_c[top], p_fp[top], 0.0))
    return out


def metrics(z_fp, z_q, alpha, K, eps, rho_c, k_max):
    """step_metrics over rows: (M [rows], c, d_loc, y, cov [rows][k_max])."""
    rows = [step_metrics(a, b, alpha, K, eps, rho_c, k_max) for a, b in zip(z_fp, z_q)]
    return (np.array([r["M"] for r in rows]), np.array([r["c"] for r in rows]),
            np.array([r["d_loc"] for r in rows]), np.array([r["y"] for r in rows]),
            np.stack([r["cov"] for r in rows]))


def calibrate_window(cov, rho_k):
    """K_b of Sec. 4.1: the smallest K whose coverage, averaged over the
    steps (rows of cov, column K - 1), reaches rho_K; 0 if no K <= k_max
    does.  Returns (K_b, mean coverage per K)."""
    mean = np.asarray(cov, dtype=np.float64).mean(axis=0)
    hit = np.nonzero(mean >= rho_k)[0]
    return (int(hit[0]) + 1 if hit.size else 0), mean
