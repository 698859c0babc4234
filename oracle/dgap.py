"""Oracle: DGAP local distribution restoration on one decode step's logits.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Follows Sec. 4.1-4.3 of the paper, in its order, all in float64:

1. features phi_t = Phi(z_hat) from the quantized logits (Sec. 4.2,
   "Runtime features");
2. detector r_t = sigmoid(f_theta(phi_t)) (Sec. 4.2, Eq. 6);
3. gate r_t > tau; r_t <= tau bypasses the corrector (Sec. 4.1, Sec. 4.3);
4. recovery window S = TopK(z_hat, K) (Sec. 4.1 Eq. 2, Sec. 4.3 Eq. 11);
5. candidate features xi_S (Sec. 4.3, "Local candidate correction");
6. corrector Delta = g_psi(xi_S, phi_t) (Sec. 4.3, Eq. 12);
7. sparse merge (Sec. 4.3, Eq. 13): z_tilde_j = z_hat_j + Delta_j for j in S
   when r_t > tau, else z_hat_j;
8. greedy token selection on z_tilde (Sec. 4.1: restoration happens before
   token selection).

Readings taken where the paper gives only categories of features or no
architecture:

* TopK orders by value descending, lowest index first among equal values;
  z_(K) (the (K+1)-th value) is also kept, for features and selection;
* phi (8 numbers): [0] entropy -sum p log p over the vocabulary, [1] top-K
  mass sum_{k<K} p_(k), [2] top-1 probability, [3] margin z_(0) - z_(1),
  [4] mean local gap (z_(0) - z_(K-1)) / (K - 1), [5] least adjacent gap
  min_k z_(k) - z_(k+1) over k < K - 1, [6] population standard deviation of
  z_(0..K-1), [7] entropy of the window distribution q = p_S / sum p_S;
* xi (5 numbers per candidate k, rank order): [0] z_(k) - z_(0),
  [1] log p_(k), [2] k / (K - 1), [3] z_(k-1) - z_(k) (0 for k = 0),
  [4] z_(k) - z_(k+1) (z_(K) for the last);
* detector: Linear(8, H) -> ReLU -> Linear(H, 1); corrector:
  [xi flattened rank-major (5K) | phi (8)] -> Linear(5K + 8, H) -> ReLU ->
  Linear(H, K); weights row-major [out][in];
* runtime temperature 1 (T appears only in the training loss, Sec. 4.3).

All of these are shift-invariant, as softmax is (Sec. 3.2).
"""

import numpy as np

N_PHI = 8
N_XI = 5


def softmax(z):
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - z.max())
    return e / e.sum()


def log_sum_exp(z):
    z = np.asarray(z, dtype=np.float64)
    m = z.max()
    return m + np.log(np.exp(z - m).sum())


def topk_window(z, K):
    """Indices of the K + 1 largest logits, value descending, lowest index
    first among equal values (a stable sort of -z)."""
    z = np.asarray(z, dtype=np.float64)
    return np.argsort(-z, kind="stable")[:K + 1]


def entropy(p):
    p = p[p > 0]
    return float(-(p * np.log(p)).sum())


def risk_features(z, K):
    """phi_t = Phi(z_hat) (Sec. 4.2).  Returns (phi [8], window [K + 1])."""
    z = np.asarray(z, dtype=np.float64)
    p = softmax(z)
    win = topk_window(z, K)
    zs = z[win[:K]]
    ps = p[win[:K]]
    mass = ps.sum()
    phi = np.array([
        entropy(p),
        mass,
        ps[0],
        zs[0] - zs[1],
        (zs[0] - zs[K - 1]) / (K - 1),
        np.min(zs[:-1] - zs[1:]),
        zs.std(),
        entropy(ps / mass),
    ])
    return phi, win


def candidate_features(z, win, K):
    """xi_{t,S} (Sec. 4.3): one row of 5 numbers per window candidate."""
    z = np.asarray(z, dtype=np.float64)
    zs = z[win[:K + 1]]  # includes z_(K)
    lse = log_sum_exp(z)
    xi = np.zeros((K, N_XI))
    for k in range(K):
        xi[k, 0] = zs[k] - zs[0]
        xi[k, 1] = zs[k] - lse
        xi[k, 2] = k / (K - 1)
        xi[k, 3] = 0.0 if k == 0 else zs[k - 1] - zs[k]
        xi[k, 4] = zs[k] - zs[k + 1]
    return xi


def mlp2(x, w1, b1, w2, b2):
    """Linear -> ReLU -> Linear, float64."""
    h = np.maximum(np.asarray(w1, np.float64) @ x + np.asarray(b1, np.float64), 0.0)
    return np.asarray(w2, np.float64) @ h + np.asarray(b2, np.float64)


def detector_logit(phi, det):
    """f_theta(phi_t) (Sec. 4.2, Eq. 6, before the sigmoid)."""
    return float(mlp2(phi, det["w1"], det["b1"], det["w2"], det["b2"])[0])


def sigmoid(f):
    return 1.0 / (1.0 + np.exp(-f))


def restore_row(z, K, tau, det, cor):
    """Run the DGAP epilogue on one row of logits (float32 in, float64 out).

    Returns a dict: idx [K] int64, z_K (the (K+1)-th value) and idx_K,
    f (detector logit), r, gate, delta [K] (zeros when not gated),
    val [K] (window values after the merge), z_tilde [V], next_token.
    """
    z = np.asarray(z, dtype=np.float64)
    if not 2 <= K < z.size:
        raise ValueError("need 2 <= K < V")
    phi, win = risk_features(z, K)
    f = detector_logit(phi, det)
    r = sigmoid(f)
    gate = bool(r > tau)
    delta = np.zeros(K)
    if gate:
        xi = candidate_features(z, win, K)
        x = np.concatenate([xi.reshape(-1), phi])
        delta = mlp2(x, cor["w1"], cor["b1"], cor["w2"], cor["b2"])
    z_tilde = z.copy()
    z_tilde[win[:K]] += delta
    return dict(idx=win[:K].copy(), idx_K=int(win[K]), z_K=z[win[K]],
                phi=phi, f=f, r=r, gate=gate, delta=delta,
                val=z_tilde[win[:K]].copy(), z_tilde=z_tilde,
                next_token=int(np.argmax(z_tilde)))


def restore(logits, K, tau, det, cor):
    """Row-wise ``restore_row`` over logits [B, V]."""
    return [restore_row(row, K, tau, det, cor) for row in np.asarray(logits)]
