"""Pins that tie the fp64 oracle to facts outside itself.

Each ``check_*`` takes an oracle module ``O`` and raises AssertionError when
the oracle disagrees with a value fixed by the paper or by mathematics:

  * closed forms: NS acting on singular values (a matrix polynomial of the
    input, Eq. (5)), geometric momentum sums (Eq. (10)), repeated decoupled
    decay (Eq. (14)), rank-one row / column RMS (Eq. (7));
  * hand values: population CV of small vectors (Eq. (8)); the Hadamard and
    diag(3, 4, 12) worked cases;
  * exact arithmetic: the NS iteration on integer matrices carried out in
    exact integers (no floating point), then the CVs and the normalisation at
    50 significant digits;
  * invariants: unit-RMS rows / columns after Eq. (9), idempotence, scale
    and sign invariance, transpose equivariance, zero rows and columns,
    and the orthogonality constraint of Section 3.1 on exact Orth;
  * paper tables: Table 5 state memory from Table 11 architectures;
  * the Muon baseline of Eq. (6): the shape factor sqrt(max(m, n)) gives an
    exactly orthogonal update unit RMS; closed forms on the Hadamard and
    known-SVD inputs.

tests/test_oracle_mutations.py plants plausible mistakes in a copy of the
oracle and asserts that at least one of these checks fails for each.
"""
from __future__ import annotations

import json
import math
import os
from fractions import Fraction

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "paper_tables.json")
A_COEF, B_COEF, C_COEF = 3.4445, -4.7750, 2.0315   # Section 2, after Eq. (5)
A_INT, B_INT, C_INT, COEF_DEN = 34445, -47750, 20315, 10000


def golden():
    with open(GOLDEN) as f:
        return json.load(f)


# ---------------------------------------------------------------- scalar forms
def p_scalar(x):
    """One quintic step on a singular value: x -> a x + b x^3 + c x^5."""
    return A_COEF * x + B_COEF * x ** 3 + C_COEF * x ** 5


def f_scalar(x, steps=5):
    for _ in range(steps):
        x = p_scalar(x)
    return x


def _orthonormal(rng, n, k):
    q, _ = np.linalg.qr(rng.standard_normal((n, k)))
    return q[:, :k]


def _sylvester_hadamard(n):
    H = np.array([[1.0]])
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]])
    return H


# ------------------------------------------------------------------ NS checks
def check_ns_known_svd(O, tol=1e-11):
    """Eq. (5) is a matrix polynomial: for H = P diag(s) Q^T, X_K = P diag(f(s/||s||)) Q^T."""
    rng = np.random.default_rng(1234)
    for (m, n, r) in [(12, 12, 12), (20, 9, 9), (7, 16, 7), (15, 11, 5), (1, 6, 1), (6, 1, 1)]:
        P = _orthonormal(rng, m, r)
        Q = _orthonormal(rng, n, r)
        s = np.exp(rng.uniform(np.log(0.05), np.log(3.0), r))
        H = P @ np.diag(s) @ Q.T
        want = P @ np.diag([f_scalar(v / np.linalg.norm(s)) for v in s]) @ Q.T
        got = O.newton_schulz(H)
        err = np.linalg.norm(got - want) / np.linalg.norm(want)
        assert err < tol, (m, n, r, err)


def check_ns_band(O):
    """Singular values of the NS output land in the band p^5 maps (x0, 1] into,
    and the singular vectors of the input are kept (Eq. (5))."""
    xs = np.linspace(3e-3, 1.0, 20001)
    fx = np.array([f_scalar(x) for x in xs])
    lo, hi = fx.min(), fx.max()
    assert 0.6 < lo < 0.75 and 1.15 < hi < 1.25, (lo, hi)
    rng = np.random.default_rng(99)
    m, n = 40, 24
    P = _orthonormal(rng, m, n)
    Q = _orthonormal(rng, n, n)
    s = np.linspace(1.0, 0.1, n)    # s / ||s|| >= 0.1 / ||s|| > 3e-3
    H = P @ np.diag(s) @ Q.T
    U = O.newton_schulz(H)
    sv = np.linalg.svd(U, compute_uv=False)
    assert sv.min() >= lo - 1e-9 and sv.max() <= hi + 1e-9, (sv.min(), sv.max())
    # singular vectors kept: P^T U Q is diagonal
    D = P.T @ U @ Q
    off = D - np.diag(np.diag(D))
    assert np.abs(off).max() < 1e-10


def check_ns_hadamard(O):
    """Worked case: H_8 (Sylvester). All singular values of H_8/||H_8||_F are
    1/sqrt(8), so X_5 = f(1/sqrt(8)) H_8 / sqrt(8); both CVs vanish, the tie
    goes to row and the normalised update is H_8 itself (entries +-1)."""
    H = _sylvester_hadamard(8)
    f = f_scalar(1.0 / math.sqrt(8.0))
    assert abs(f - 1.066967948) < 5e-9, f
    U = O.newton_schulz(H)
    assert np.abs(U - f * H / math.sqrt(8.0)).max() < 1e-13
    Ut, info = O.equilibrate_hidden(U)
    assert info["gamma_r"] < 1e-12 and info["gamma_c"] < 1e-12
    assert info["direction"] == O.ROW
    assert np.abs(Ut - H).max() < 1e-12


def check_ns_diag_4x3(O):
    """Worked case: H = [diag(3, 4, 12); 0] (||H||_F = 13). NS acts on each
    diagonal entry: U = [diag(f(3/13), f(4/13), f(12/13)); 0]. The zero row is
    excluded from gamma_r; gamma_r = gamma_c exactly, so row is chosen and
    the update is sqrt(3) [I_3; 0] (column normalisation would give 2 [I_3; 0])."""
    H = np.zeros((4, 3))
    H[0, 0], H[1, 1], H[2, 2] = 3.0, 4.0, 12.0
    U = O.newton_schulz(H)
    want = np.zeros((4, 3))
    for i, v in enumerate((3, 4, 12)):
        want[i, i] = f_scalar(v / 13.0)
    assert np.abs(U - want).max() < 1e-13
    Ut, info = O.equilibrate_hidden(U)
    assert abs(info["gamma_r"] - info["gamma_c"]) < 1e-12
    assert info["direction"] == O.ROW
    exp = np.zeros((4, 3))
    exp[:3, :3] = math.sqrt(3.0) * np.eye(3)
    assert np.abs(Ut - exp).max() < 1e-12
    # the column reading, forced, gives 2 [I; 0]
    Utc, _ = O.equilibrate_hidden(U, force_direction=O.COL)
    exp[:3, :3] = 2.0 * np.eye(3)
    assert np.abs(Utc - exp).max() < 1e-12


def check_ns_zero_rows_cols(O):
    """Zero rows / columns of the input stay exactly zero through Eq. (5) and
    are excluded from the CVs of Eq. (8)."""
    rng = np.random.default_rng(5)
    H = rng.standard_normal((9, 7))
    H[2, :] = 0.0
    H[:, 4] = 0.0
    U = O.newton_schulz(H)
    assert np.all(U[2, :] == 0.0) and np.all(U[:, 4] == 0.0)
    r, c = O.row_col_rms(U)
    keep_r = np.delete(r, 2)
    m = keep_r.mean()
    want = math.sqrt(((keep_r - m) ** 2).mean()) / m
    assert abs(O.coefficient_of_variation(r) - want) < 1e-12
    Ut, _ = O.equilibrate_hidden(U)
    assert np.all(Ut[2, :] == 0.0) and np.all(Ut[:, 4] == 0.0)
    assert np.all(O.newton_schulz(np.zeros((3, 5))) == 0.0)


# ------------------------------------------------------ exact integer NS
def _imat(M, N):
    return [[sum(M[i][k] * N[k][j] for k in range(len(N))) for j in range(len(N[0]))] for i in range(len(M))]


def _itrans(M):
    return [list(r) for r in zip(*M)]


def exact_ns(H_int, steps=5):
    """Eq. (5) in exact integers: X_k = M_k / D_k, X_0 = H / ||H||_F with an
    integer norm. One step gives
      M' = a' M D^4 + b' (M M^T) M D^2 + c' (M M^T)^2 M,   D' = 10^4 D^5
    with (a', b', c') = 10^4 (a, b, c) integers."""
    N2 = sum(v * v for row in H_int for v in row)
    N = math.isqrt(N2)
    assert N * N == N2
    M, D = [list(r) for r in H_int], N
    for _ in range(steps):
        G = _imat(M, _itrans(M))
        GM = _imat(G, M)
        GGM = _imat(G, GM)
        D2 = D * D
        D4 = D2 * D2
        M = [[A_INT * M[i][j] * D4 + B_INT * GM[i][j] * D2 + C_INT * GGM[i][j]
              for j in range(len(M[0]))] for i in range(len(M))]
        D = COEF_DEN * D4 * D
    return M, D


def _integer_matrix_with_integer_norm(rng, m, n, lo=-6, hi=7):
    while True:
        H = rng.integers(lo, hi, size=(m, n))
        s = int((H * H).sum())
        if s > 0 and math.isqrt(s) ** 2 == s:
            return [[int(v) for v in row] for row in H]


def check_ns_exact_integer(O):
    """Oracle NS == exact rational NS on integer 4x3 and 8x8 inputs, and the
    CVs, direction and normalised update == a 50-digit evaluation."""
    mpmath = __import__("mpmath")
    mp = mpmath.mp
    mp.dps = 50
    rng = np.random.default_rng(2024)
    for (m, n) in [(4, 3), (8, 8), (3, 5)]:
        H = _integer_matrix_with_integer_norm(rng, m, n)
        M, D = exact_ns(H)
        exact = np.array([[float(Fraction(v, D)) for v in row] for row in M])
        got = O.newton_schulz(np.array(H, dtype=np.float64))
        assert np.abs(got - exact).max() <= 1e-13 * np.abs(exact).max(), (m, n)
        U = [[mpmath.mpf(v) / D for v in row] for row in M]
        r = [mpmath.sqrt(sum(x * x for x in row) / n) for row in U]
        c = [mpmath.sqrt(sum(U[i][j] ** 2 for i in range(m)) / m) for j in range(n)]

        def cv(v):
            v = [x for x in v if x > mpmath.mpf("1e-7")]
            mu = sum(v) / len(v)
            return mpmath.sqrt(sum((x - mu) ** 2 for x in v) / len(v)) / mu
        gr, gc = cv(r), cv(c)
        Ut, info = O.equilibrate_hidden(got)
        assert abs(info["gamma_r"] - float(gr)) < 1e-12 and abs(info["gamma_c"] - float(gc)) < 1e-12
        d = 0 if gr >= gc else 1
        if abs(gr - gc) > 1e-6:
            assert info["direction"] == d
        if info["direction"] == 0:
            want = [[float(U[i][j] / r[i]) for j in range(n)] for i in range(m)]
        else:
            want = [[float(U[i][j] / c[j]) for j in range(n)] for i in range(m)]
        assert np.abs(Ut - np.array(want)).max() < 1e-12


# ------------------------------------------------------ stats / normalisation
def check_row_col_rms_rank_one(O):
    """Eq. (7) on u v^T: r_i = |u_i| ||v|| / sqrt(n), c_j = |v_j| ||u|| / sqrt(m)."""
    rng = np.random.default_rng(7)
    u = rng.standard_normal(6)
    v = rng.standard_normal(11)
    r, c = O.row_col_rms(np.outer(u, v))
    assert np.allclose(r, np.abs(u) * np.linalg.norm(v) / math.sqrt(11), rtol=1e-14, atol=0)
    assert np.allclose(c, np.abs(v) * np.linalg.norm(u) / math.sqrt(6), rtol=1e-14, atol=0)


def check_cv_hand_values(O):
    """Eq. (8): population std / mean over entries above delta."""
    assert abs(O.coefficient_of_variation([1.0, 3.0]) - 0.5) < 1e-15
    assert abs(O.coefficient_of_variation([0.0, 1.0, 3.0]) - 0.5) < 1e-15
    assert abs(O.coefficient_of_variation([1e-7, 1.0, 3.0]) - 0.5) < 1e-15     # at delta: excluded
    assert abs(O.coefficient_of_variation([2.0, 4.0, 4.0, 4.0, 5.0, 5.0, 7.0, 9.0]) - 0.4) < 1e-15
    assert O.coefficient_of_variation([0.0, 0.0]) == 0.0
    assert O.coefficient_of_variation([2.5, 2.5, 2.5]) == 0.0
    # scale invariance (Section 3.1)
    v = np.array([0.3, 1.7, 2.2, 0.9])
    assert abs(O.coefficient_of_variation(v) - O.coefficient_of_variation(1e3 * v)) < 1e-14


def check_selection_rule(O):
    """Eq. (11): row when gamma_r >= gamma_c, column otherwise."""
    assert O.select_direction(0.5, 0.1) == O.ROW
    assert O.select_direction(0.1, 0.5) == O.COL
    assert O.select_direction(0.3, 0.3) == O.ROW
    rng = np.random.default_rng(11)
    # a matrix with strong row imbalance and equal column norms chooses row
    X = rng.standard_normal((30, 30))
    X = X / np.linalg.norm(X, axis=0, keepdims=True)        # unit columns
    X = X * np.linspace(0.2, 3.0, 30)[:, None]              # then rows scaled
    r, c = O.row_col_rms(X)
    assert O.coefficient_of_variation(r) > O.coefficient_of_variation(c)
    _, info = O.equilibrate_hidden(X)
    assert info["direction"] == O.ROW
    _, info = O.equilibrate_hidden(X.T)
    assert info["direction"] == O.COL


def check_equilibration_invariants(O):
    """Eq. (9): every nonzero row (column) gets unit RMS; the chosen side's CV
    is 0; N_r is idempotent; the update is invariant to positive scaling and
    odd in the input (Sections 3.1-3.2)."""
    rng = np.random.default_rng(3)
    X = rng.standard_normal((13, 21)) * np.exp(rng.uniform(-2, 2, 13))[:, None]
    X[4, :] = 0.0
    Nr = O.row_normalize(X)
    rr = np.sqrt((Nr ** 2).sum(1) / 21)
    assert np.allclose(np.delete(rr, 4), 1.0, atol=1e-14) and rr[4] == 0.0
    assert abs((Nr ** 2).sum() - 12 * 21) < 1e-10           # ||.||_F^2 = m_+ n
    assert np.abs(O.row_normalize(Nr) - Nr).max() < 1e-14   # idempotent
    Nc = O.col_normalize(X)
    cc = np.sqrt((Nc ** 2).sum(0) / 13)
    assert np.allclose(cc, 1.0, atol=1e-14)
    assert abs((Nc ** 2).sum() - 21 * 13) < 1e-10
    # rows scaled by 1/r_i: check one entry by hand
    r4 = math.sqrt((X[5] ** 2).sum() / 21)
    assert abs(Nr[5, 7] - X[5, 7] / r4) < 1e-14
    c3 = math.sqrt((X[:, 3] ** 2).sum() / 13)
    assert abs(Nc[8, 3] - X[8, 3] / c3) < 1e-14
    Ut, info = O.equilibrate_hidden(X)
    side = info["direction"]
    r2, c2 = O.row_col_rms(Ut)
    assert O.coefficient_of_variation(r2 if side == O.ROW else c2) < 1e-12
    # whole step: scale and sign invariance, transpose equivariance
    B = rng.standard_normal((10, 16)) * np.exp(rng.uniform(-1, 1, 16))[None, :]
    U1, i1 = O.equilibrate_hidden(O.newton_schulz(B))
    U2, i2 = O.equilibrate_hidden(O.newton_schulz(37.5 * B))
    U3, i3 = O.equilibrate_hidden(O.newton_schulz(-B))
    U4, i4 = O.equilibrate_hidden(O.newton_schulz(B.T))
    assert i1["direction"] == i2["direction"] == i3["direction"]
    assert np.abs(U1 - U2).max() < 1e-11 and np.abs(U1 + U3).max() < 1e-11
    assert i4["direction"] != i1["direction"] and np.abs(U1 - U4.T).max() < 1e-11


def check_rms_threshold_scale_zero(O):
    """Reading of Eq. (9) (the paper rescales only nonzero rows / columns and
    sets delta for Eq. (8)): a row or column whose RMS does not exceed delta
    gets scale 0, in N_r, N_c, both stages of Eq. (12) and Eq. (13), while
    one just above delta is rescaled to unit RMS like any other."""
    rng = np.random.default_rng(14)
    X = rng.standard_normal((6, 10))
    X[2] = 5e-8 * np.sign(rng.standard_normal(10))      # RMS 5e-8 <= delta
    X[3] = 3e-7 * np.sign(rng.standard_normal(10))      # RMS 3e-7 > delta
    Nr = O.row_normalize(X)
    assert np.all(Nr[2] == 0.0)
    assert abs(math.sqrt((Nr[3] ** 2).mean()) - 1.0) < 1e-12 and abs(Nr[3, 0] - X[3, 0] / 3e-7) < 1e-6
    Nc = O.col_normalize(X.T)
    assert np.all(Nc[:, 2] == 0.0) and abs(math.sqrt((Nc[:, 3] ** 2).mean()) - 1.0) < 1e-12
    # Eq. (12): the small row is dropped by N_r, so it is zero after N_c too;
    # a column that is tiny in every row is dropped by the second stage
    B = rng.standard_normal((7, 5))
    B[4] = 2e-8
    B[:, 1] = 1e-12
    T = O.two_sided_normalize(B)
    assert np.all(T[4] == 0.0)
    Rn = O.row_normalize(B)
    c1 = math.sqrt((Rn[:, 1] ** 2).mean())
    assert 0.0 < c1 <= O.DELTA and np.all(T[:, 1] == 0.0)
    # Eq. (13): a vector with RMS <= delta is not rescaled
    assert np.all(O.vector_normalize(np.full(9, 4e-8)) == 0.0)
    w = O.vector_normalize(np.full(9, -2e-7))
    assert np.allclose(w, -1.0, atol=1e-12)


def check_orthogonality_constraint(O):
    """Section 3.1: exact Orth of a tall full-rank matrix has Y^T Y = I, so
    gamma_c = 0 and row is chosen; a wide one has gamma_r = 0 and picks column."""
    rng = np.random.default_rng(8)
    Htall = rng.standard_normal((40, 12)) * np.exp(rng.uniform(-1, 1, 40))[:, None]
    P, _, Qt = np.linalg.svd(Htall, full_matrices=False)
    Y = P @ Qt
    r, c = O.row_col_rms(Y)
    assert O.coefficient_of_variation(c) < 1e-12 and O.coefficient_of_variation(r) > 0.05
    _, info = O.equilibrate_hidden(Y)
    assert info["direction"] == O.ROW
    _, info = O.equilibrate_hidden(Y.T)
    assert info["direction"] == O.COL


def check_two_sided_and_vector(O):
    """Eq. (12): after N_c(N_r(B)) every nonzero column has unit RMS; Eq. (13):
    the vector update has unit RMS."""
    rng = np.random.default_rng(4)
    B = rng.standard_normal((17, 9)) * np.exp(rng.uniform(-2, 2, 17))[:, None]
    T = O.two_sided_normalize(B)
    assert np.allclose(np.sqrt((T ** 2).sum(0) / 17), 1.0, atol=1e-14)
    Rn = B / np.sqrt((B ** 2).sum(1, keepdims=True) / 9)
    assert np.abs(T - Rn / np.sqrt((Rn ** 2).sum(0, keepdims=True) / 17)).max() < 1e-13
    v = rng.standard_normal(33) * 5.0
    w = O.vector_normalize(v)
    assert abs(math.sqrt((w ** 2).mean()) - 1.0) < 1e-14
    assert abs(w[3] - v[3] / math.sqrt((v ** 2).mean())) < 1e-14


def check_param_step_branches(O):
    """Algorithm 1's three branches: a vector's update has RMS 1 (Eq. (13));
    a remaining 2D parameter's update has unit-RMS columns (Eq. (12)); a
    hidden weight goes through NS (its Hadamard case gives H_8)."""
    rng = np.random.default_rng(21)
    lr, mu, wd = 0.02, 0.95, 0.1
    v = rng.standard_normal(40) * 3.0
    Wn, B, Ut = O.param_step(O.VECTOR, np.zeros(40), v, np.zeros(40), lr, mu, wd)
    assert np.abs(B - v).max() == 0.0 and abs(math.sqrt((Ut ** 2).mean()) - 1.0) < 1e-14
    assert np.abs(Wn + 0.2 * lr * v / math.sqrt((v ** 2).mean())).max() < 1e-15
    M = rng.standard_normal((30, 12)) * np.exp(rng.uniform(-2, 2, 30))[:, None]
    Wn, B, Ut = O.param_step(O.REMAINING_2D, np.zeros((30, 12)), M, np.zeros((30, 12)), lr, mu, wd)
    assert np.allclose(np.sqrt((Ut ** 2).sum(0) / 30), 1.0, atol=1e-14)
    H = _sylvester_hadamard(8)
    _, _, Ut = O.param_step(O.HIDDEN, np.zeros((8, 8)), H, np.zeros((8, 8)), lr, mu, wd)
    assert np.abs(Ut - H).max() < 1e-12


# ------------------------------------------------------------- momentum / apply
def check_momentum_closed_form(O):
    """Eq. (10) with a constant gradient: B_t = G (1 - mu^(t+1)) / (1 - mu)."""
    rng = np.random.default_rng(6)
    G = rng.standard_normal((5, 4))
    mu = 0.95
    B = np.zeros_like(G)
    for t in range(12):
        B = O.momentum_update(B, G, mu)
        assert np.abs(B - G * (1 - mu ** (t + 1)) / (1 - mu)).max() < 1e-12
    # Nesterov look-ahead input: G + mu * B_t
    Bp = rng.standard_normal((5, 4))
    Bt = O.momentum_update(Bp, G, mu)
    assert np.abs(O.ns_input(Bt, G, mu, nesterov=True) - (G + mu * (mu * Bp + G))).max() < 1e-14
    assert np.abs(O.ns_input(Bt, G, mu, nesterov=False) - (mu * Bp + G)).max() < 1e-14


def check_apply_closed_form(O):
    """Eq. (14) repeated with a fixed update V:
    W_t = q^t W_0 - rho eta V (1 - q^t) / (1 - q),  q = 1 - eta lambda."""
    rng = np.random.default_rng(10)
    W0 = rng.standard_normal((3, 7))
    V = rng.standard_normal((3, 7))
    lr, wd, rho = 0.02, 0.1, 0.2
    q = 1 - lr * wd
    W = W0
    for t in range(1, 9):
        W = O.apply_update(W, V, lr, wd, rho)
        assert np.abs(W - (q ** t * W0 - rho * lr * V * (1 - q ** t) / (1 - q))).max() < 1e-13
    # one hand value
    assert abs(O.apply_update(np.array([1.0]), np.array([2.0]), 0.5, 0.1, 0.2)[0] - (0.95 - 0.2)) < 1e-15


def check_hidden_step_composition(O):
    """Algorithm 1, hidden branch: one step from B_{-1} = 0 on the Hadamard
    gradient gives W_1 = (1 - eta lambda) W_0 - rho eta H_8."""
    H = _sylvester_hadamard(8)
    W0 = np.arange(64, dtype=np.float64).reshape(8, 8) / 100.0
    W1, B, info = O.hidden_step(W0, H, np.zeros((8, 8)), lr=0.02, mu=0.95, weight_decay=0.1)
    assert np.abs(B - H).max() == 0.0
    assert np.abs(W1 - ((1 - 0.002) * W0 - 0.2 * 0.02 * H)).max() < 1e-14


def check_moonlight_update(O):
    """Eq. (6): sqrt(max(m, n)) makes the update RMS independent of the shape.
    For U with orthonormal rows (m <= n) or columns (m > n), ||U||_F^2 =
    min(m, n), so the applied update (W_{t+1} - (1 - eta lambda) W_t) /
    (eta rho) has RMS exactly 1; decay is decoupled."""
    rng = np.random.default_rng(31)
    lr, wd, rho = 0.02, 0.1, 0.2
    for m, n in [(12, 30), (30, 12), (16, 16), (1, 9), (9, 1)]:
        U = _orthonormal(rng, max(m, n), min(m, n))
        U = U.T if m < n else U
        assert U.shape == (m, n)
        W0 = rng.standard_normal((m, n))
        V = (O.moonlight_update(W0, U, lr, wd, rho) - (1 - lr * wd) * W0) / (-lr * rho)
        assert abs(np.sqrt((V * V).mean()) - 1.0) < 1e-12, (m, n)
        assert np.abs(V - np.sqrt(max(m, n)) * U).max() < 1e-12
    # no update and no decay: identity
    W0 = rng.standard_normal((4, 5))
    assert np.abs(O.moonlight_update(W0, np.zeros((4, 5)), lr, 0.0, rho) - W0).max() == 0.0


def check_moonlight_step(O):
    """Eq. (6) composed with Eqs. (10) and (5), from B_{-1} = 0.
    Hadamard gradient: U = f(1/sqrt 8) H_8 / sqrt 8, so the update is
    -eta rho f(1/sqrt 8) H_8 (MeqMuon's would be -eta rho H_8: the factor f is
    what equilibration removes). Known SVD, rectangular: U = P f(s/||s||) Q^T
    and the update is -eta rho sqrt(max(m, n)) U."""
    lr, mu, wd, rho = 0.02, 0.95, 0.1, 0.2
    H = _sylvester_hadamard(8)
    W0 = np.arange(64, dtype=np.float64).reshape(8, 8) / 100.0
    W1, B, U = O.moonlight_step(W0, H, np.zeros((8, 8)), lr, mu, wd, rho)
    f = f_scalar(1.0 / math.sqrt(8.0))
    assert np.abs(B - H).max() == 0.0
    assert np.abs(W1 - ((1 - lr * wd) * W0 - lr * rho * f * H)).max() < 1e-13
    rng = np.random.default_rng(77)
    for m, n in [(10, 26), (26, 10)]:
        r = min(m, n)
        P = _orthonormal(rng, m, r)
        Q = _orthonormal(rng, n, r)
        sv = np.exp(rng.uniform(np.log(0.1), np.log(2.0), r))
        G = P @ np.diag(sv) @ Q.T
        Uk = P @ np.diag([f_scalar(v / np.linalg.norm(sv)) for v in sv]) @ Q.T
        W1, _, _ = O.moonlight_step(np.zeros((m, n)), G, np.zeros((m, n)), lr, mu, wd, rho)
        assert np.abs(W1 + lr * rho * np.sqrt(max(m, n)) * Uk).max() < 1e-12, (m, n)
    # Nesterov: the NS input is G_t + mu B_t
    Bp = rng.standard_normal((6, 9))
    G = rng.standard_normal((6, 9))
    _, _, U = O.moonlight_step(np.zeros((6, 9)), G, Bp, lr, mu, wd, rho, nesterov=True)
    Bt = mu * Bp + G
    assert np.abs(U - O.newton_schulz(G + mu * Bt)).max() < 1e-13


def check_ns_cv_trajectory(O):
    """Section 3.1 replay of Eq. (5). diag(3, 4, 12) with a zero row: every
    iterate is [diag(f_k(3/13), f_k(4/13), f_k(12/13)); 0], so both CVs at k
    are the population CV of the three scalar iterates (the zero row is
    excluded). Rank one u v^T: every iterate is a multiple of u v^T, so the
    trajectory is flat at (CV|u|, CV|v|). The last point is the CVs of the
    K-step NS output, and the trajectory is scale-free."""
    H = np.zeros((4, 3))
    H[0, 0], H[1, 1], H[2, 2] = 3.0, 4.0, 12.0
    gr, gc = O.ns_cv_trajectory(H, steps=20)
    assert len(gr) == len(gc) == 21
    x = np.array([3.0, 4.0, 12.0]) / 13.0
    for k in range(21):
        cv = np.std(x) / np.mean(x)
        assert abs(gr[k] - cv) < 1e-12 and abs(gc[k] - cv) < 1e-12, (k, gr[k], gc[k], cv)
        x = np.array([p_scalar(v) for v in x])
    rng = np.random.default_rng(41)
    u = rng.uniform(0.5, 2.0, 9) * rng.choice([-1.0, 1.0], 9)
    v = rng.uniform(0.1, 3.0, 14) * rng.choice([-1.0, 1.0], 14)
    gr, gc = O.ns_cv_trajectory(np.outer(u, v), steps=12)
    cvu = np.std(np.abs(u)) / np.mean(np.abs(u))
    cvv = np.std(np.abs(v)) / np.mean(np.abs(v))
    assert np.abs(gr - cvu).max() < 1e-12 and np.abs(gc - cvv).max() < 1e-12
    G = rng.standard_normal((10, 17)) * rng.uniform(0.1, 5.0, 10)[:, None]
    gr, gc = O.ns_cv_trajectory(G, steps=5)
    r5, c5 = O.row_col_rms(O.newton_schulz(G, steps=5))
    assert abs(gr[5] - O.coefficient_of_variation(r5)) < 1e-12
    assert abs(gc[5] - O.coefficient_of_variation(c5)) < 1e-12
    gr2, gc2 = O.ns_cv_trajectory(1024.0 * G, steps=5)
    assert np.abs(gr2 - gr).max() < 1e-12 and np.abs(gc2 - gc).max() < 1e-12


# ------------------------------------------------------------ paper tables
def llama_hidden_counts(a):
    q = a["q_heads"] * a["head_dim"]
    kv = a["kv_heads"] * a["head_dim"]
    d, f, L = a["hidden"], a["ffn"], a["layers"]
    Nh = L * (q * d + 2 * kv * d + d * q + 3 * d * f)
    Rh = L * (q + 2 * kv + d + 2 * f + d)
    return Nh, Rh


def check_state_memory_table(O=None):
    """Table 5 from Table 11: Muon = N_h + 2 N_a, NorMuon = + R_h, MeqMuon =
    N_h + N_a values of 4 bytes (Section 4, 'Memory overhead')."""
    g = golden()
    for name, a in g["architecture"].items():
        Nh, Rh = llama_hidden_counts(a)
        Na = a["params_m"] * 1e6 - Nh
        mib = lambda x: round(4 * x / 2 ** 20, 2)
        assert mib(Nh + 2 * Na) == g["state_mib"]["Muon"][name], name
        assert mib(Nh + 2 * Na + Rh) == g["state_mib"]["NorMuon"][name], name
        assert mib(Nh + Na) == g["state_mib"]["MeqMuon"][name], name


def check_constants(O):
    g = golden()
    assert tuple(O.NS_COEFFS) == (g["ns"]["a"], g["ns"]["b"], g["ns"]["c"])
    assert O.NS_STEPS == g["ns"]["steps"] and O.DELTA == g["delta"] and O.RHO == g["rho"]


ALL_CHECKS = [
    check_constants, check_ns_known_svd, check_ns_band, check_ns_hadamard, check_ns_diag_4x3,
    check_ns_zero_rows_cols, check_ns_exact_integer, check_row_col_rms_rank_one,
    check_cv_hand_values, check_selection_rule, check_equilibration_invariants, check_rms_threshold_scale_zero,
    check_orthogonality_constraint, check_two_sided_and_vector, check_momentum_closed_form,
    check_apply_closed_form, check_hidden_step_composition, check_param_step_branches,
    check_moonlight_update, check_moonlight_step, check_ns_cv_trajectory,
]
