"""Plain fp64 CPU oracle for the MeqMuon optimizer step (hidden-layer 2D weights).

TEST INFRASTRUCTURE ONLY. Nothing in the product path may import this module:
only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` use it. It shares no code with the
CUDA path and the CUDA path never calls it.

It follows the paper ("MeqMuon: Matrix-Equilibrating Muon for LLM
Pretraining") step by step, in the paper's notation, with numpy float64 and
``numpy.matmul`` as the only library primitive. There is no blocking, fusion,
reordering or shape trick (no transposition of tall matrices, no symmetric
Gram shortcut): each function is the equation it cites, written out.

Equation numbers are the paper's:
  Eq. (5)  quintic Newton-Schulz iteration           (Section 2, "Muon");
           its row / column CV trajectory               (Section 3.1)
  Eq. (6)  Muon with decoupled weight decay and RMS
           alignment (the Moonlight form), the baseline
           MeqMuon is compared with                   (Section 2, "Muon")
  Eq. (7)  row / column RMS vectors                  (Section 3.1)
  Eq. (8)  coefficients of variation, delta rule     (Section 3.1)
  Eq. (9)  row / column normalisation operators      (Section 3.2)
  Eq. (10) momentum                                  (Section 3.2)
  Eq. (11) adaptive one-sided selection              (Section 3.2)
  Eq. (12) two-sided normalisation                   (Section 3.2)
  Eq. (13) 1D global-RMS normalisation               (Section 3.2)
  Algorithm 1, all three parameter branches          (param_step)
  Eq. (14) parameter update with decoupled decay     (Section 3.2)
  Algorithm 1 (MeqMuon), hidden-weight branch        (Section 3.2)

Readings of points the paper leaves open, each with the reason stated:
  * Zero input to NS: the paper defines the iteration for a nonzero input
    only (Section 2); a zero momentum matrix gives U = 0.
  * A row / column RMS that does not exceed delta counts as zero
    (Section 3.1): they are excluded from the CVs and their normalisation
    scale is 0, so they contribute no update.
  * Ties in Eq. (11): row is chosen when gamma_r >= gamma_c - tie_atol, with
    tie_atol = 1e-6 (an absolute tolerance on the dimensionless CVs) so that
    ties that are exact in real arithmetic do not depend on rounding order.
    tie_atol = 0 gives the literal ">=" rule.
  * Nesterov momentum (Section 4 says the experiments used it, with no
    formula): when enabled, the NS input is G_t + mu * B_t; otherwise it is
    B_t as in Eq. (10) and Algorithm 1.
"""
from __future__ import annotations

import numpy as np

# (a, b, c) and K of the quintic iteration, Section 2 (after Eq. (5)) and
# Section 4 (5 iterations with these coefficients).
NS_COEFFS = (3.4445, -4.7750, 2.0315)
NS_STEPS = 5
# RMS threshold delta of Section 3.1 (an RMS that does not exceed it counts as zero).
DELTA = 1e-7
# RMS alignment coefficient rho, Section 4.
RHO = 0.2
TIE_ATOL = 1e-6

ROW = 0
COL = 1


def _f64(x):
    return np.asarray(x, dtype=np.float64)


def momentum_update(B_prev, G, mu):
    """Eq. (10): B_t = mu * B_{t-1} + G_t, with B_{-1} = 0 (Algorithm 1)."""
    return mu * _f64(B_prev) + _f64(G)


def ns_input(B, G, mu, nesterov=False):
    """Matrix that is orthogonalised. Eq. (10) / Algorithm 1 feed B_t itself.

    With ``nesterov`` (Section 4 names Nesterov momentum for the experiments
    without a formula) the input is the look-ahead G_t + mu * B_t.
    """
    B = _f64(B)
    if nesterov:
        return _f64(G) + mu * B
    return B


def newton_schulz(H, steps=NS_STEPS, coeffs=NS_COEFFS):
    """Eq. (5): X_0 = H / ||H||_F; A_k = X_k X_k^T; X_{k+1} = a X_k + (b A_k + c A_k^2) X_k.

    Returns X_K. The literal orientation of Eq. (5) is kept for every shape
    (A_k is m x m even when m > n). A zero H returns zeros (reading above).
    """
    a, b, c = coeffs
    H = _f64(H)
    nrm = np.sqrt(np.sum(H * H))
    if nrm == 0.0:
        return np.zeros_like(H)
    X = H / nrm
    for _ in range(steps):
        A = np.matmul(X, X.T)
        AA = np.matmul(A, A)
        X = a * X + np.matmul(b * A + c * AA, X)
    return X


def ns_cv_trajectory(H, steps=20, coeffs=NS_COEFFS, delta=DELTA):
    """Eq. (8) CVs of the row and column RMS (Eq. (7)) of every iterate of
    Eq. (5), k = 0..steps (Section 3.1 replays the NS iteration this way on
    saved pre-NS matrices). Returns (gamma_r, gamma_c), each of length
    steps + 1; a zero H gives zeros."""
    a, b, c = coeffs
    H = _f64(H)
    nrm = np.sqrt(np.sum(H * H))
    gr, gc = [], []
    X = H / nrm if nrm > 0.0 else np.zeros_like(H)
    for k in range(steps + 1):
        r, cc = row_col_rms(X)
        gr.append(coefficient_of_variation(r, delta))
        gc.append(coefficient_of_variation(cc, delta))
        if k < steps:
            A = np.matmul(X, X.T)
            X = a * X + np.matmul(b * A + c * np.matmul(A, A), X)
    return np.array(gr), np.array(gc)


def row_col_rms(X):
    """Eq. (7): r_i = ||X_{i,:}||_2 / sqrt(n), c_j = ||X_{:,j}||_2 / sqrt(m)."""
    X = _f64(X)
    m, n = X.shape
    r = np.sqrt(np.sum(X * X, axis=1)) / np.sqrt(n)
    c = np.sqrt(np.sum(X * X, axis=0)) / np.sqrt(m)
    return r, c


def coefficient_of_variation(v, delta=DELTA):
    """Eq. (8): population standard deviation over mean, taken over the
    entries greater than delta (zero rows / columns are excluded, Section 3.1).
    With no such entry the CV is 0."""
    v = _f64(v)
    keep = v[v > delta]
    if keep.size == 0:
        return 0.0
    mean = np.sum(keep) / keep.size
    var = np.sum((keep - mean) ** 2) / keep.size
    return float(np.sqrt(var) / mean)


def select_direction(gamma_r, gamma_c, tie_atol=TIE_ATOL):
    """Eq. (11): row-wise when gamma_r >= gamma_c, else column-wise (ties,
    within tie_atol, go to row)."""
    return ROW if gamma_r >= gamma_c - tie_atol else COL


def _inverse_rms(v, delta):
    v = _f64(v)
    out = np.zeros_like(v)
    nz = v > delta
    out[nz] = 1.0 / v[nz]
    return out


def row_normalize(X, delta=DELTA):
    """Eq. (9): N_r(X) = diag(r^{-1}) X; rows with r_i <= delta get scale 0."""
    r, _ = row_col_rms(X)
    return _inverse_rms(r, delta)[:, None] * _f64(X)


def col_normalize(X, delta=DELTA):
    """Eq. (9): N_c(X) = X diag(c^{-1}); columns with c_j <= delta get scale 0."""
    _, c = row_col_rms(X)
    return _f64(X) * _inverse_rms(c, delta)[None, :]


def equilibrate_hidden(U, delta=DELTA, force_direction=None, tie_atol=TIE_ATOL):
    """Eq. (11): pick N_r or N_c for the orthogonalised update U.

    Returns (U_tilde, info) where info holds r, c, gamma_r, gamma_c and the
    chosen direction. ``force_direction`` (ROW / COL) overrides the choice
    (used to compare against a run that chose the other side of a near-tie).
    """
    r, c = row_col_rms(U)
    gr = coefficient_of_variation(r, delta)
    gc = coefficient_of_variation(c, delta)
    d = select_direction(gr, gc, tie_atol) if force_direction is None else force_direction
    Ut = row_normalize(U, delta) if d == ROW else col_normalize(U, delta)
    return Ut, {"r": r, "c": c, "gamma_r": gr, "gamma_c": gc, "direction": d}


def two_sided_normalize(B, delta=DELTA):
    """Eq. (12): N_c(N_r(B)) for the remaining 2D parameters."""
    return col_normalize(row_normalize(B, delta), delta)


def vector_normalize(b, delta=DELTA):
    """Eq. (13): B / (||B||_2 / sqrt(d)) for 1D parameters (zero if the RMS is
    at or below delta, the same reading as for rows and columns)."""
    b = _f64(b)
    rms = np.sqrt(np.sum(b * b)) / np.sqrt(b.size)
    if rms <= delta:
        return np.zeros_like(b)
    return b / rms


def apply_update(W, U_tilde, lr, weight_decay, rho=RHO):
    """Eq. (14): W_{t+1} = (1 - eta_t lambda) W_t - rho eta_t U_tilde."""
    return (1.0 - lr * weight_decay) * _f64(W) - rho * lr * _f64(U_tilde)


def hidden_step(W, G, B_prev, lr, mu, weight_decay, eps=DELTA, rho=RHO,
                steps=NS_STEPS, coeffs=NS_COEFFS, nesterov=False,
                force_direction=None, tie_atol=TIE_ATOL):
    """Algorithm 1, branch for a 2D weight in a hidden layer, for one matrix.

    Returns (W_next, B_t, info); info also carries U (the NS output) and
    U_tilde (the normalised update).
    """
    B = momentum_update(B_prev, G, mu)
    U = newton_schulz(ns_input(B, G, mu, nesterov), steps, coeffs)
    Ut, info = equilibrate_hidden(U, eps, force_direction, tie_atol)
    W_next = apply_update(W, Ut, lr, weight_decay, rho)
    info = dict(info, U=U, U_tilde=Ut)
    return W_next, B, info


HIDDEN = 0          # 2D weight in a hidden layer
REMAINING_2D = 1    # remaining 2D parameter (token embedding, LM head)
VECTOR = 2          # 1D parameter (RMSNorm weight, bias)


def param_step(kind, W, G, B_prev, lr, mu, weight_decay, eps=DELTA, rho=RHO, **kw):
    """Algorithm 1 for one parameter of any type: Eq. (10) momentum, then the
    normalised update of its branch (Eq. (11) after Eq. (5) for hidden 2D
    weights, Eq. (12) for the remaining 2D parameters, Eq. (13) for 1D
    parameters), then Eq. (14). Returns (W_next, B_t, U_tilde)."""
    if kind == HIDDEN:
        Wn, B, info = hidden_step(W, G, B_prev, lr, mu, weight_decay, eps=eps, rho=rho, **kw)
        return Wn, B, info["U_tilde"]
    B = momentum_update(B_prev, G, mu)
    if kind == REMAINING_2D:
        Ut = two_sided_normalize(B, eps)
    elif kind == VECTOR:
        Ut = vector_normalize(B, eps)
    else:
        raise ValueError(kind)
    return apply_update(W, Ut, lr, weight_decay, rho), B, Ut


def moonlight_update(W, U, lr, weight_decay, rho=RHO):
    """Eq. (6): W_{t+1} = (1 - eta_t lambda) W_t - eta_t rho sqrt(max(m, n)) U_t.
    sqrt(max(m, n)) compensates the update RMS for the matrix shape."""
    m, n = np.shape(U)
    return (1.0 - lr * weight_decay) * _f64(W) - lr * rho * np.sqrt(max(m, n)) * _f64(U)


def moonlight_step(W, G, B_prev, lr, mu, weight_decay, rho=RHO, steps=NS_STEPS, coeffs=NS_COEFFS,
                   nesterov=False):
    """Eq. (6) for one 2D weight in a hidden layer: Eq. (10) momentum, Orth
    approximated by the K iterations of Eq. (5), then the shape-compensated
    update, with no equilibration. Returns (W_next, B_t, U_t)."""
    B = momentum_update(B_prev, G, mu)
    U = newton_schulz(ns_input(B, G, mu, nesterov), steps, coeffs)
    return moonlight_update(W, U, lr, weight_decay, rho), B, U


def hidden_step_all(Ws, Gs, Bs_prev, lr, mu, weight_decay, **kw):
    """Algorithm 1 over a list of hidden matrices (each handled independently;
    the direction is chosen per matrix, Section 3.2)."""
    out_W, out_B, infos = [], [], []
    for W, G, Bp in zip(Ws, Gs, Bs_prev):
        Wn, B, info = hidden_step(W, G, Bp, lr, mu, weight_decay, **kw)
        out_W.append(Wn)
        out_B.append(B)
        infos.append(info)
    return out_W, out_B, infos
