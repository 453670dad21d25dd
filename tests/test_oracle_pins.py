"""Pins for the CPU oracle: hand-worked fixtures, closed forms, exact invariants, library
routines and brute force.  None of them reuses the oracle's own formula to check itself."""
import os

from fractions import Fraction

import numpy as np
import pytest
import scipy.linalg

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed=0):
    return np.random.default_rng(seed)


def _rand_spd(rng, k, cond=10.0):
    Q, _ = np.linalg.qr(rng.standard_normal((k, k)))
    lam = np.exp(rng.uniform(0, np.log(cond), k))
    return (Q * lam) @ Q.T


def _rand_orth(rng, d):
    Q, R = np.linalg.qr(rng.standard_normal((d, d)))
    return Q * np.sign(np.diag(R))


# ------------------------------------------------------------------------------------------
# Quantizer (Lemma 2 range, App. A.2.1 steps, Sec. 6 RTN)
# ------------------------------------------------------------------------------------------

def _read_quant_golden():
    cases = []
    with open(os.path.join(GOLDEN, "quantizer_rows.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            row, s, codes = [p.strip() for p in line.split("|")]
            # a step written as a fraction "a/7" is compared with its correctly rounded float64 value
            num, _, den = s.partition("/")
            s_val = float(Fraction(num) / Fraction(den or "1"))
            cases.append((np.array([float(v) for v in row.split()]), s_val,
                          np.array([int(v) for v in codes.split()])))
    return cases


@pytest.mark.parametrize("case", range(8))
def test_quantizer_hand_worked_rows(case):
    row, s_exp, q_exp = _read_quant_golden()[case]
    q, s, pre = O.quantize_rows_symmetric(row[None, :])
    assert s[0] == s_exp
    np.testing.assert_array_equal(q[0], q_exp)


def test_quantizer_golden_covers_ties_that_float32_breaks_the_wrong_way():
    """The tie rows are chosen so that deciding the code as rint(f32(v) * f32(7 / a)) gives a
    different code than the definition: the fixture can tell the two apart."""
    diff = 0
    for row, _, q_exp in _read_quant_golden():
        a = np.float32(np.max(np.abs(row)))
        if a == 0:
            continue
        q32 = np.rint(row.astype(np.float32) * (np.float32(7) / a)).astype(np.int64)
        diff += int(np.sum(q32 != q_exp))
    assert diff >= 3


def test_quantizer_ranges_and_error_bound():
    rng = _rng(1)
    V = rng.standard_normal((200, 96)) * np.exp(rng.standard_normal((200, 1)))
    V[3] = 0.0
    V[7, 5] = 40.0  # an outlier
    q, s, pre = O.quantize_rows_symmetric(V)
    assert q.min() >= -7 and q.max() <= 7
    # the element of largest magnitude maps to +-7
    idx = np.argmax(np.abs(V), axis=1)
    big = q[np.arange(V.shape[0]), idx]
    assert np.all(np.abs(big[np.arange(200) != 3]) == 7)
    # zero row
    assert s[3] == 0 and np.all(q[3] == 0)
    # |v - s q| <= s / 2 (no clipping: the range covers the row)
    err = np.abs(V - q * s[:, None])
    assert np.all(err <= s[:, None] / 2 * (1 + 1e-12) + 1e-300)
    # away from rounding boundaries the code is the round-to-nearest of v / s
    far = (np.abs(np.abs(pre) - np.floor(np.abs(pre)) - 0.5) > 1e-9) & (s[:, None] > 0)
    np.testing.assert_array_equal(q[far], np.rint(V[far] / np.repeat(s[:, None], V.shape[1], 1)[far]))
    # step size is max|v| / 7 exactly
    np.testing.assert_array_equal(s, np.max(np.abs(V), axis=1) / 7)


def test_quantizer_bit_widths():
    rng = _rng(2)
    V = rng.standard_normal((50, 33))
    for b in (2, 3, 4, 6, 8):
        q, s, _ = O.quantize_rows_symmetric(V, bits=b)
        qmax = 2 ** (b - 1) - 1
        assert q.min() == -qmax or q.max() == qmax
        assert np.abs(q).max() == qmax


# ------------------------------------------------------------------------------------------
# Hadamard, matrix powers and the geometric mean (Sec. 4, Eq. 7)
# ------------------------------------------------------------------------------------------

def test_hadamard_matches_textbook_order4_and_is_orthonormal():
    H4 = np.loadtxt(os.path.join(GOLDEN, "hadamard4.txt"))
    np.testing.assert_array_equal(O.hadamard(4) * 2.0, H4)
    for k in (1, 2, 32, 128, 256):
        H = O.hadamard(k)
        np.testing.assert_allclose(H @ H.T, np.eye(k), atol=1e-12)
        np.testing.assert_allclose(np.abs(H), 1 / np.sqrt(k), rtol=1e-14)
    with pytest.raises(ValueError):
        O.hadamard(12)


def test_spd_power_against_scipy_sqrtm_and_inverse():
    rng = _rng(3)
    A = _rand_spd(rng, 24, cond=1e4)
    np.testing.assert_allclose(O.spd_power(A, 0.5), scipy.linalg.sqrtm(A).real, rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(O.spd_power(A, -1.0), np.linalg.inv(A), rtol=1e-8, atol=1e-12)
    with pytest.raises(np.linalg.LinAlgError):
        O.spd_power(-np.eye(3), 0.5)


def test_geometric_mean_closed_forms_and_riccati():
    rng = _rng(4)
    # scalars: a # b = sqrt(a b)
    assert np.isclose(O.geometric_mean(np.array([[4.0]]), np.array([[9.0]]))[0, 0], 6.0, rtol=1e-14)
    # commuting (diagonal) matrices: A # B = (A B)^{1/2}
    a, b = rng.uniform(0.1, 10, 7), rng.uniform(0.1, 10, 7)
    np.testing.assert_allclose(O.geometric_mean(np.diag(a), np.diag(b)), np.diag(np.sqrt(a * b)), rtol=1e-12)
    # general SPD: G = A # B is the SPD solution of G A^{-1} G = B, symmetric in A, B, and A # A^{-1} = I
    A, B = _rand_spd(rng, 16, 1e3), _rand_spd(rng, 16, 1e3)
    G = O.geometric_mean(A, B)
    np.testing.assert_allclose(G @ np.linalg.inv(A) @ G, B, rtol=1e-8, atol=1e-10)
    np.testing.assert_allclose(G, O.geometric_mean(B, A), rtol=1e-8, atol=1e-10)
    assert np.linalg.eigvalsh(G).min() > 0
    np.testing.assert_allclose(O.geometric_mean(A, np.linalg.inv(A)), np.eye(16), atol=1e-9)


def test_alignment_optimal_M_fixed_point_eq8():
    """Eq. 8: M Sigma_x M = M^{-1} Sigma_w M^{-1}; its eigenvalues are those of
    (Sigma_x^{1/2} Sigma_w Sigma_x^{1/2})^{1/2} (the printed right-hand side is garbled)."""
    rng = _rng(5)
    Sx, Sw = _rand_spd(rng, 12, 1e3), _rand_spd(rng, 12, 1e2)
    M, Mi = O.alignment_optimal_M(Sx, Sw)
    np.testing.assert_allclose(M @ Mi, np.eye(12), atol=1e-9)
    L = M @ Sx @ M
    np.testing.assert_allclose(L, Mi @ Sw @ Mi, rtol=1e-8, atol=1e-10)
    # eigenvalues
    Sxh = scipy.linalg.sqrtm(Sx).real
    ref = np.sqrt(np.linalg.eigvalsh(Sxh @ Sw @ Sxh))
    np.testing.assert_allclose(np.sort(np.linalg.eigvalsh(L)), np.sort(ref), rtol=1e-8)
    # and Sigma_w = G Sigma_x G with G = M^2 (definition of Sigma_w # Sigma_x^{-1})
    np.testing.assert_allclose(M @ M @ Sx @ M @ M, Sw, rtol=1e-8, atol=1e-10)


# ------------------------------------------------------------------------------------------
# Calibration statistics and brute force
# ------------------------------------------------------------------------------------------

def test_calib_cov_blocks_brute_force():
    rng = _rng(6)
    X = rng.standard_normal((37, 24))
    S = O.calib_cov_block_sums(X, 8)
    full = np.zeros((24, 24))
    for t in range(37):  # one outer product per token
        full += np.outer(X[t], X[t])
    for b in range(3):
        np.testing.assert_allclose(S[b], full[b * 8:(b + 1) * 8, b * 8:(b + 1) * 8], rtol=1e-13)
    W = rng.standard_normal((19, 24))
    Sw = O.weight_autocorr_blocks(W, 8)
    WtW = W.T @ W
    for b in range(3):
        np.testing.assert_allclose(Sw[b], WtW[b * 8:(b + 1) * 8, b * 8:(b + 1) * 8], rtol=1e-13)


def test_int_gemm_brute_force_and_extremes():
    rng = _rng(7)
    qx = rng.integers(-7, 8, (9, 70))
    qw = rng.integers(-7, 8, (5, 70))
    acc = O.int_gemm(qx, qw)
    for t in range(9):
        for o in range(5):
            assert acc[t, o] == sum(int(qx[t, i]) * int(qw[o, i]) for i in range(70))
    # largest accumulator of the layers here: 49 * 14336
    big = O.int_gemm(np.full((2, 14336), 7), np.full((3, 14336), -7))
    assert np.all(big == -49 * 14336)
    assert acc.dtype == np.int64


def test_dequantize_output_orientation():
    acc = np.array([[1, 2, 3], [4, 5, 6]])
    y = O.dequantize_output(acc, np.array([2.0, 3.0]), np.array([1.0, 10.0, 100.0]))
    np.testing.assert_array_equal(y, [[2, 40, 600], [12, 150, 1800]])


def test_sqnr_hand_worked():
    vals = dict(l.split() for l in open(os.path.join(GOLDEN, "sqnr_example.txt")) if l[0] != "#")
    y = np.array([[1.0, 2.0], [3.0, 4.0]])
    yh = np.array([[1.0, 2.0], [3.0, 3.0]])
    sig, err = O.sqnr_sums(y, yh)
    assert sig == float(vals["sig"]) and err == float(vals["err"])
    assert abs(O.sqnr_db(y, yh) - float(vals["sqnr_db"])) < 1e-12
    assert abs(O.sqnr_db(np.ones(10), 0.9 * np.ones(10)) - 20.0) < 1e-9


# ------------------------------------------------------------------------------------------
# Transforms: function preservation (Eq. 5), rotation invariance (Eq. 4)
# ------------------------------------------------------------------------------------------

@pytest.mark.parametrize("kind", ["identity", "rht", "cat"])
def test_function_preservation_eq5(kind):
    rng = _rng(8)
    d, k = 64, 16
    X = rng.standard_normal((300, d)) @ rng.standard_normal((d, d)) * 0.3
    X[:, 5] *= 40
    W = rng.standard_normal((48, d)) * 0.02
    signs = rng.choice([-1.0, 1.0], d)
    Sx = O.calib_cov_block_sums(X, k) / X.shape[0]
    Sw = O.weight_autocorr_blocks(W, k)
    T, Ti = O.build_transform(kind, d, k, Sx, Sw, signs)
    for b in range(d // k):
        np.testing.assert_allclose(T[b] @ Ti[b], np.eye(k), atol=1e-9)
    y = O.linear(X, W)
    y2 = O.linear(O.apply_act_transform(X, T), O.apply_weight_transform(W, Ti))
    assert np.linalg.norm(y2 - y) / np.linalg.norm(y) < 1e-10


def test_act_transform_is_T_times_x():
    rng = _rng(9)
    d, k = 12, 4
    T = rng.standard_normal((3, k, k))
    X = rng.standard_normal((5, d))
    Tfull = scipy.linalg.block_diag(*T)
    np.testing.assert_allclose(O.apply_act_transform(X, T), (Tfull @ X.T).T, rtol=1e-13)
    Ti = rng.standard_normal((3, k, k))
    W = rng.standard_normal((7, d))
    np.testing.assert_allclose(O.apply_weight_transform(W, Ti), W @ scipy.linalg.block_diag(*Ti), rtol=1e-13)


def test_rht_signs_and_alignment_invariance_eq4():
    rng = _rng(10)
    d, k = 32, 8
    X = rng.standard_normal((500, d)) * rng.uniform(0.1, 5, d)
    W = rng.standard_normal((20, d))
    signs = rng.choice([-1.0, 1.0], d)
    T, Ti = O.build_transform("rht", d, k, signs=signs)
    H = O.hadamard(k)
    np.testing.assert_allclose(T[1], H @ np.diag(signs[k:2 * k]), rtol=1e-14)
    a0 = O.alignment(X, W)
    a1 = O.alignment(O.apply_act_transform(X, T), O.apply_weight_transform(W, Ti))
    assert abs(a1 - a0) < 1e-12 * a0
    R = _rand_orth(rng, d)
    a2 = O.alignment(X @ R.T, W @ R.T)
    assert abs(a2 - a0) < 1e-12 * a0


def test_alignment_moment_form_and_bound():
    rng = _rng(11)
    X = rng.standard_normal((400, 16)) * rng.uniform(0.1, 3, 16)
    W = rng.standard_normal((10, 16))
    a = O.alignment(X, W)
    assert abs(a - O.alignment_from_moments(X.T @ X / 400, W.T @ W)) < 1e-12
    assert 0 < a <= 1.0


# ------------------------------------------------------------------------------------------
# Optimal alignment (Eq. 7, Eq. 9), block optimality (Eq. 10) and k = 1
# ------------------------------------------------------------------------------------------

def test_full_rank_M_reaches_max_alignment_eq9_and_beats_random():
    rng = _rng(12)
    d = 10
    X = rng.standard_normal((2000, d)) @ rng.standard_normal((d, d))
    W = rng.standard_normal((14, d)) * rng.uniform(0.2, 3, (14, 1))
    Sx, Sw = X.T @ X / X.shape[0], W.T @ W
    M, Mi = O.alignment_optimal_M(Sx, Sw)
    a_opt = O.alignment(X @ M.T, W @ Mi)
    a_max = O.max_alignment(Sx, W)
    # closed form written independently: singular values of W Sigma_x^{1/2}
    sv = np.linalg.svd(W @ scipy.linalg.sqrtm(Sx).real, compute_uv=False)
    assert abs(a_max - np.sum(sv ** 2) / np.sum(sv) ** 2) < 1e-8 * a_max
    assert abs(a_opt - a_max) < 1e-7 * a_max
    assert a_opt > O.alignment(X, W)
    for _ in range(1500):
        Mr = rng.standard_normal((d, d)) + 3 * np.eye(d) * rng.uniform(0, 1)
        Mr2 = M @ (np.eye(d) + 0.05 * rng.standard_normal((d, d)))
        for MM in (Mr, Mr2):
            if abs(np.linalg.det(MM)) < 1e-6:
                continue
            assert O.alignment(X @ MM.T, W @ np.linalg.inv(MM)) <= a_opt * (1 + 1e-9)


def _blocks_data(rng, d, n=3000):
    X = rng.standard_normal((n, d)) @ rng.standard_normal((d, d)) * 0.5
    X[:, 3] *= 30
    W = rng.standard_normal((2 * d, d)) * rng.lognormal(0, 0.5, (2 * d, 1))
    return X, W


def test_block_cat_is_optimal_among_block_diagonal_transforms():
    """Eq. 10: solving each k x k block on its own sub-problem is optimal among all block-diagonal
    transforms (no per-block rescaling raises alignment), with closed form
    A = Tr(Sw Sx) / (sum_b Tr((Sx_b^{1/2} Sw_b Sx_b^{1/2})^{1/2}))^2."""
    rng = _rng(13)
    d, k = 16, 4
    X, W = _blocks_data(rng, d)
    Sx_full = X.T @ X / X.shape[0]
    Sxb = O.calib_cov_block_sums(X, k) / X.shape[0]
    Swb = O.weight_autocorr_blocks(W, k)
    T, Ti = O.build_transform("cat", d, k, Sxb, Swb)
    a_cat = O.alignment(O.apply_act_transform(X, T), O.apply_weight_transform(W, Ti))
    denom = 0.0
    for b in range(d // k):
        h = scipy.linalg.sqrtm(Sxb[b]).real
        denom += np.trace(scipy.linalg.sqrtm(h @ Swb[b] @ h).real)
    closed = np.trace(W.T @ W @ Sx_full) / denom ** 2
    assert abs(a_cat - closed) < 1e-9 * closed
    assert a_cat >= O.alignment(X, W)
    assert a_cat <= O.max_alignment(Sx_full, W) * (1 + 1e-12)
    for _ in range(300):
        c = np.exp(rng.standard_normal(d // k))
        D = np.repeat(c, k)
        Ts = T * c[:, None, None]
        Tis = Ti / c[:, None, None]
        assert O.alignment(O.apply_act_transform(X, Ts), O.apply_weight_transform(W, Tis)) <= a_cat * (1 + 1e-10)
        Rb = rng.standard_normal((d // k, k, k)) + 2 * np.eye(k)
        Rbi = np.linalg.inv(Rb)
        assert O.alignment(O.apply_act_transform(X, Rb), O.apply_weight_transform(W, Rbi)) <= a_cat * (1 + 1e-10)
        del D


def test_k1_closed_form_diagonal_scaling():
    """End of Sec. 4: for k = 1 the block solution is a diagonal scaling; from Eq. 7 with 1 x 1
    blocks m_i = (sum_j W_ji^2 / E[x_i^2])^{1/4} (the printed exponent is garbled)."""
    rng = _rng(14)
    d = 12
    X, W = _blocks_data(rng, d)
    Sxb = O.calib_cov_block_sums(X, 1) / X.shape[0]
    Swb = O.weight_autocorr_blocks(W, 1)
    T, Ti = O.build_transform("cat", d, 1, Sxb, Swb)
    m = (np.sum(W ** 2, axis=0) / np.mean(X ** 2, axis=0)) ** 0.25
    np.testing.assert_allclose(T[:, 0, 0], m, rtol=1e-12)
    a = O.alignment(X * m, W / m)
    for i in range(d):  # finite-difference perturbations never raise A
        for eps in (1e-3, -1e-3, 0.1, -0.1):
            mm = m.copy()
            mm[i] *= np.exp(eps)
            assert O.alignment(X * mm, W / mm) <= a * (1 + 1e-12)


# ------------------------------------------------------------------------------------------
# SQNR decomposition (App. A.1 and A.2): exact identities, then the approximations
# ------------------------------------------------------------------------------------------

def test_error_expansion_identity_app_a1():
    rng = _rng(15)
    X = rng.standard_normal((256, 32)) * rng.uniform(0.2, 4, 32)
    W = rng.standard_normal((24, 32)) * 0.1
    qx, sx, _ = O.quantize_rows_symmetric(X)
    qw, sw, _ = O.quantize_rows_symmetric(W)
    Xq, Wq = O.dequantize_rows(qx, sx), O.dequantize_rows(qw, sw)
    dX, dW = X - Xq, W - Wq
    sig, err = O.sqnr_sums(O.linear(X, W), O.linear(Xq, Wq))
    a = np.sum((dX @ W.T) ** 2)
    b = np.sum((X @ dW.T) ** 2)
    c = np.sum((dX @ dW.T) ** 2)
    cross = 2 * (np.sum((dX @ W.T) * (X @ dW.T)) - np.sum((dX @ W.T) * (dX @ dW.T))
                 - np.sum((X @ dW.T) * (dX @ dW.T)))
    assert abs(err - (a + b + c + cross)) < 1e-10 * err
    assert abs(sig - np.sum((X @ W.T) ** 2)) < 1e-10 * sig
    # acc-based path equals the dequantized float path
    _, yh = O.w4a4_linear(qx, sx, qw, sw)
    np.testing.assert_allclose(yh, O.linear(Xq, Wq), rtol=1e-12, atol=1e-14)


def test_activation_mse_trace_form_app_a21():
    """App. A.2.1: E||W dx||^2 = Tr(W^T W E[dx dx^T]) exactly."""
    rng = _rng(16)
    X = rng.standard_normal((500, 20))
    W = rng.standard_normal((9, 20))
    q, s, _ = O.quantize_rows_symmetric(X)
    dX = X - O.dequantize_rows(q, s)
    lhs = np.mean(np.sum((dX @ W.T) ** 2, axis=1))
    rhs = np.trace(W.T @ W @ (dX.T @ dX / 500))
    assert abs(lhs - rhs) < 1e-12 * lhs


def test_concentration_bounds():
    """Sec. 2 (Concentration): lowest value 1/4 (-6 dB) for symmetric, 1/2 (-3 dB) for asymmetric."""
    onehot = np.zeros((3, 10))
    onehot[np.arange(3), [1, 4, 9]] = [2.0, -5.0, 0.5]
    assert O.concentration_act(onehot) == 0.25
    pair = np.zeros((2, 8))
    pair[:, 0], pair[:, 1] = 3.0, -3.0
    assert O.concentration_act(pair, symmetric=False) == 0.5
    rng = _rng(17)
    for _ in range(20):
        V = rng.standard_normal((50, 16)) ** 3
        assert O.concentration_act(V) >= 0.25
        assert O.concentration_act(V, symmetric=False) >= 0.5
        assert O.concentration_weight(V) >= 0.25
    # scale invariance (Sec. 2)
    V = rng.standard_normal((30, 12))
    assert abs(O.concentration_act(V * 7.5) - O.concentration_act(V)) < 1e-14


def test_weight_concentration_closed_forms():
    """Sec. 2, Lemma 3: C(W) = sum_o ||w_o||^2 / sum_o (2 max_i |w_oi|)^2 over output rows.  Rows
    of equal magnitudes c in d entries give d c^2 / (4 c^2) = d / 4; one-hot rows give 1/4; a
    mix weights each row by its squared range (a ratio of sums, not a mean of ratios)."""
    d = 12
    flat = np.where(np.arange(3 * d).reshape(3, d) % 2 == 0, 1.0, -1.0) * np.array([[0.5], [2.0], [3.0]])
    assert O.concentration_weight(flat) == d / 4
    onehot = np.zeros((4, d))
    onehot[np.arange(4), [0, 3, 7, 11]] = [1.0, -2.0, 0.25, 9.0]
    assert O.concentration_weight(onehot) == 0.25
    mix = np.vstack([flat[:1], onehot[:1] * 0.5])   # ||.||^2 = 12 * 0.25 and 0.25; ranges 1 and 1
    assert abs(O.concentration_weight(mix) - (3.0 + 0.25) / (1.0 + 1.0)) < 1e-15


def test_lemmas_and_theorem1_on_gaussian_layer():
    """Lemma 1-3 / Theorem 1 are approximations; the paper reports them accurate between 5 and
    50 dB (Sec. 2).  On a Gaussian layer: within 0.2 dB at 8 bits, 1 dB at 4 bits, and about
    6 dB per extra bit (Eq. 3)."""
    rng = _rng(18)
    d = 64
    X = rng.standard_normal((60000, d))
    W = rng.standard_normal((64, d))
    for bits, tol in ((8, 0.2), (4, 1.0)):
        ma = O.sqnr_act_only(X, W, bits)
        mw = O.sqnr_weight_only(X, W, bits)
        mb = O.sqnr_both(X, W, bits, bits)
        assert abs(O.db(O.lemma2_act_sqnr(X, W, bits)) - O.db(ma)) < tol
        assert abs(O.db(O.lemma3_weight_sqnr(X, W, bits)) - O.db(mw)) < tol
        assert abs(O.db(O.parallel(ma, mw)) - O.db(mb)) < tol          # Lemma 1
        assert abs(O.db(O.theorem1_sqnr(X, W, bits, bits)) - O.db(mb)) < tol
    g = O.db(O.sqnr_both(X, W, 10, 10)) - O.db(O.sqnr_both(X, W, 9, 9))
    assert 5.8 < g < 6.3


def test_identity_transform_is_plain_rtn():
    rng = _rng(19)
    X = rng.standard_normal((40, 32)) * 3
    W = rng.standard_normal((16, 32))
    out = O.cat_layer(X, W, "identity", 8)
    qx, sx, _ = O.quantize_rows_symmetric(X)
    qw, sw, _ = O.quantize_rows_symmetric(W)
    np.testing.assert_array_equal(out["act"].qx, qx)
    np.testing.assert_array_equal(out["prep"].qw, qw)
    np.testing.assert_array_equal(out["acc"], O.int_gemm(qx, qw))


def test_cat_improves_sqnr_on_outlier_layer():
    """Sec. 4 / Fig. 6 (qualitative): CAT raises alignment and SQNR over no transform and over a
    randomized Hadamard rotation on a layer with correlated channels and outliers."""
    import workloads as WL
    cfg = WL.small_config("pin", d_in=256, d_out=192, n_eval=512, n_calib=512, k=32, dtype="f32", seed=3)
    L = WL.make_layer(cfg)
    X, W, Xc = L.x_eval.values, L.W.values, L.x_calib.values
    res = {kind: O.cat_layer(X, W, kind, cfg.k, X_calib=Xc, signs=L.rht_signs) for kind in ("identity", "rht", "cat")}
    assert res["rht"]["sqnr_db"] > res["identity"]["sqnr_db"]
    assert res["cat"]["sqnr_db"] > res["rht"]["sqnr_db"]
    for r in res.values():
        assert np.linalg.norm(r["prep"].Wt @ np.eye(256)) > 0


# ------------------------------------------------------------------------------------------
# Asymmetric per-token quantizer (Sec. 6 set-up; Lemma 2 asymmetric range)
# ------------------------------------------------------------------------------------------

def _read_asym_golden():
    cases = []
    with open(os.path.join(GOLDEN, "quantizer_asym_rows.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            bits, row, s, z, codes = [p.strip() for p in line.split("|")]
            num, _, den = s.partition("/")
            cases.append((int(bits), np.array([float(v) for v in row.split()]), float(Fraction(num) / Fraction(den or "1")),
                          int(z), np.array([int(v) for v in codes.split()])))
    return cases


@pytest.mark.parametrize("case", range(6))
def test_asymmetric_quantizer_hand_worked_rows(case):
    bits, row, s_exp, z_exp, q_exp = _read_asym_golden()[case]
    q, s, z, pre = O.quantize_rows_asymmetric(row[None, :], bits)
    assert s[0] == s_exp and z[0] == z_exp
    np.testing.assert_array_equal(q[0], q_exp)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_asymmetric_quantizer_range_and_error_bound(bits):
    rng = _rng(40 + bits)
    V = rng.standard_normal((300, 77)) * np.exp(rng.standard_normal((300, 1)))
    V[5] = np.abs(V[5]) + 1.0            # all positive (ReLU-like)
    V[6] = -np.abs(V[6])                 # all non-positive
    V[7] = 0.0
    N = 2 ** bits - 1
    q, s, z, pre = O.quantize_rows_asymmetric(V, bits)
    assert q.min() >= 0 and q.max() <= N
    Qv = O.dequantize_rows_asymmetric(q, s, z)
    # every value of the (zero-including) range is within half a step: no clipping
    assert np.all(np.abs(V - Qv) <= s[:, None] / 2 * (1 + 1e-12) + 1e-300)
    # zero is on the grid, and the extremes of a row use the extreme codes
    assert np.all((z >= 0) & (z <= N))
    np.testing.assert_array_equal(O.dequantize_rows_asymmetric(z[:, None], s, z), 0.0)
    pos, neg = V.max(axis=1) > 0, V.min(axis=1) < 0
    assert np.all(q[pos].max(axis=1) == N) and np.all(q[neg].min(axis=1) == 0)
    assert s[7] == 0 and np.all(q[7] == 0)
    # the step is the asymmetric range over N intervals (Lemma 2), the range taken with zero
    lo, hi = np.minimum(V.min(axis=1), 0), np.maximum(V.max(axis=1), 0)
    np.testing.assert_allclose(s, (hi - lo) / N, rtol=1e-15)


def test_asymmetric_beats_symmetric_on_shifted_data_only():
    """Sec. 2 (Concentration): asymmetric quantization helps a lot for shifted data (after a ReLU)
    and little for zero-centred data.  Here on the activation side of a layer at 4 bits."""
    rng = _rng(44)
    W = rng.standard_normal((64, 96)) * 0.05
    Xc = rng.standard_normal((4000, 96))             # zero-centred
    Xr = np.maximum(Xc, 0.0) + 0.05                  # shifted, one-sided
    def act_sqnr(X, asym):
        if asym:
            q, s, z, _ = O.quantize_rows_asymmetric(X, 4)
            Xq = O.dequantize_rows_asymmetric(q, s, z)
        else:
            q, s, _ = O.quantize_rows_symmetric(X, 4)
            Xq = O.dequantize_rows(q, s)
        return O.sqnr_db(O.linear(X, W), O.linear(Xq, W))
    assert abs(act_sqnr(Xc, True) - act_sqnr(Xc, False)) < 1.5
    assert act_sqnr(Xr, True) > act_sqnr(Xr, False) + 4.0


# ------------------------------------------------------------------------------------------
# L_2.4 weight range search (Sec. 6, following GPTQ)
# ------------------------------------------------------------------------------------------

def test_weight_range_search_properties():
    rng = _rng(45)
    W = rng.standard_normal((50, 128)) * 0.02
    W[3, 7] = 2.0                                   # one outlier 100x the rest: clipping it would cost more
    W[4] = 0.0                                      # zero row: every candidate scores 0 -> the full range
    W[5] = np.repeat([-7.0, -3.0, 0.0, 2.0, 7.0], 26)[:128] * 0.125   # every value on the full range's grid
    i = O.weight_range_lp(W, 4)
    assert i.shape == (50,) and np.all((i >= 0) & (i < 80))
    assert i[4] == 0 and i[5] == 0                  # zero error at the full range: the first minimum
    # the chosen range never scores worse than the full range (it is a candidate)
    def score(row, shrink, bits=4, p=2.4):
        qmax = 2 ** (bits - 1) - 1
        s = (100 - shrink) / 100 * np.max(np.abs(row)) / qmax
        q = np.clip(np.round(row / s), -qmax, qmax) if s > 0 else 0 * row
        return np.sum(np.abs(row - q * s) ** p)
    for r in range(50):
        if r == 4:
            continue
        assert score(W[r], i[r]) <= score(W[r], 0) * (1 + 1e-12)
    # Gaussian rows at 4 bits clip (the L_2.4 optimum lies inside the max range); the outlier row keeps
    # its full range (clipping the outlier costs more than rounding the small values to zero)
    assert np.median(i[6:]) > 0 and i[3] == 0
    # scale invariance: a power-of-two scale of a row leaves the chosen range
    np.testing.assert_array_equal(O.weight_range_lp(W * 8.0, 4), i)
    # codes at the chosen range are clamped to the grid, and the step is the shrunk range over qmax
    q, s, _ = O.quantize_rows_symmetric(W, 4, shrink=i)
    assert q.min() >= -7 and q.max() <= 7
    assert q[3, 7] == 7 and np.all(q[3, np.arange(128) != 7] == 0)
    np.testing.assert_allclose(s, np.max(np.abs(W), axis=1) * (100 - i) / 100 / 7, rtol=1e-15)


def test_shrunk_range_ties_are_exact():
    """With a shrunk range a_i = max|w| (100 - i) / 100 the quotient qmax v / a_i is evaluated from
    exact operands, (700 v) / (max|w| (100 - i)), so a value exactly half-way between two points of the
    shrunk grid rounds to even.  Hand-worked: max|w| = 1, i = 30 (a_i = 0.7, step 0.1): v = 0.25 is
    2.5 steps -> 2, v = -0.25 -> -2, v = 0.35 (not a binary fraction) ~ 3.5 steps -> by the float64
    quotient of the stored value; v = 0.75 is 7.5 steps -> clamped to 7."""
    q, s, pre = O.quantize_rows_symmetric(np.array([[1.0, 0.25, -0.25, 0.75, 0.0]]), 4, shrink=np.array([30]))
    assert pre[0, 1] == 2.5 and pre[0, 2] == -2.5 and pre[0, 3] == 7.5
    np.testing.assert_array_equal(q[0], [7, 2, -2, 7, 0])
    assert s[0] == 0.7 / 7
    # the same values at i = 0 (full range, step 1/7): 7 * 0.25 = 1.75 -> 2, 0.75 -> 5.25 -> 5
    q0, _, _ = O.quantize_rows_symmetric(np.array([[1.0, 0.25, -0.25, 0.75, 0.0]]), 4, shrink=np.array([0]))
    np.testing.assert_array_equal(q0[0], [7, 2, -2, 5, 0])


def test_l24_range_improves_weight_sqnr_at_4_bits():
    """Weight-only SQNR with the L_2.4 range is at least that of the max range (Sec. 6 uses it)."""
    rng = _rng(46)
    W = rng.standard_t(5, (256, 128)) * 0.02
    X = rng.standard_normal((2000, 128))
    def w_sqnr(shrink):
        q, s, _ = O.quantize_rows_symmetric(W, 4, shrink=shrink)
        return O.sqnr_db(O.linear(X, W), O.linear(X, O.dequantize_rows(q, s)))
    assert w_sqnr(O.weight_range_lp(W, 4)) >= w_sqnr(None) + 0.5


# ------------------------------------------------------------------------------------------
# Bit widths of the whole layer (Sec. 2: ~6 dB per bit; Fig. 1, Fig. 6: W4A4 vs W6A6)
# ------------------------------------------------------------------------------------------

def test_layer_bit_widths_gain_about_6db_per_bit():
    rng = _rng(47)
    X = rng.standard_normal((3000, 64))
    W = rng.standard_normal((48, 64)) * 0.05
    sq = {b: O.cat_layer(X, W, "identity", 32, bits_x=b, bits_w=b)["sqnr_db"] for b in (4, 6, 8)}
    assert 10.5 < sq[6] - sq[4] < 13.5
    assert 10.5 < sq[8] - sq[6] < 13.5
    w4a8 = O.cat_layer(X, W, "identity", 32, bits_x=8, bits_w=4)["sqnr_db"]
    assert sq[4] < w4a8 < sq[8]


def test_layer_asymmetric_accumulators_match_dequantized_product():
    """With asymmetric activations the integer path sum (q_x - z) q_w times the steps equals the
    product of the dequantized operands (Sec. 3, Eq. 5)."""
    rng = _rng(48)
    X = rng.standard_normal((70, 64)) + 0.7
    W = rng.standard_normal((33, 64)) * 0.1
    r = O.cat_layer(X, W, "identity", 16, bits_x=4, bits_w=4, act_asym=True, w_range="l2.4")
    ac, pw = r["act"], r["prep"]
    Xq = O.dequantize_rows_asymmetric(ac.qx, ac.sx, ac.zx)
    Wq = O.dequantize_rows(pw.qw, pw.sw)
    np.testing.assert_allclose(r["y_hat"], Xq @ Wq.T, rtol=1e-12, atol=1e-12)


def test_interval_count_of_the_grid_is_measured_by_the_noise():
    """N in Lemmas 2-3 is the number of quantization intervals across the range r = 2 max|v|: the
    noise variance is s^2 / 12 with s = r / N.  On dense rows (the noise is uniform) the measured
    r / sqrt(12 E[e^2]) is 2 qmax = 14 at 4 bits on the restricted grid used here, not the paper's
    2^b - 1 = 15 -- n_intervals must return the grid's count (and 2 at 2 bits, 254 at 8 bits)."""
    rng = _rng(60)
    V = rng.uniform(-1, 1, (4000, 512))
    V[:, 0] = 1.0                                    # every row's range is exactly 2
    for bits in (2, 3, 4, 8):
        q, s, _ = O.quantize_rows_symmetric(V, bits)
        e = V[:, 1:] - q[:, 1:] * s[:, None]
        n_meas = 2.0 / np.sqrt(12 * np.mean(e * e))
        assert abs(n_meas / O.n_intervals(bits) - 1) < 0.01, (bits, n_meas)
        assert abs(n_meas / O.n_intervals(bits, paper=True) - 1) > 0.05 or bits == 8


# ------------------------------------------------------------------------------------------
# Full-size Hadamard and the alignment ceiling (Sec. 4: T = H M_hat; Eq. 9)
# ------------------------------------------------------------------------------------------

def test_full_size_hadamard_keeps_alignment_and_function():
    """Composing the block M_hat with the full-size H_d changes concentration only: A(T x, W T^{-1})
    equals A(M_hat x, W M_hat^{-1}) exactly (alignment is rotation invariant, Sec. 2 Eq. 4 / Sec. 4),
    and (W T^{-1})(T x) = W x (Eq. 5)."""
    rng = _rng(70)
    d, k = 64, 16
    X = rng.standard_normal((600, d)) @ (rng.standard_normal((d, d)) * 0.3 + np.eye(d))
    X[:, 5] *= 30.0
    W = rng.standard_normal((40, d)) * 0.05
    Sx = O.calib_cov_block_sums(X, k) / X.shape[0]
    Sw = O.weight_autocorr_blocks(W, k)
    T, Ti, M, Mi = O.build_transform_full_hadamard(d, k, Sx, Sw)
    np.testing.assert_allclose(T @ Ti, np.eye(d), atol=1e-10)
    np.testing.assert_allclose((W @ Ti) @ (X @ T.T).T, W @ X.T, rtol=1e-9, atol=1e-9)
    Mb, Mib = O.block_diag(M), O.block_diag(Mi)
    assert abs(O.alignment(X @ T.T, W @ Ti) / O.alignment(X @ Mb.T, W @ Mib) - 1) < 1e-12
    # the block-H_k variant has the same alignment too (its rotation is block-diagonal)
    Tk, Tik = O.build_transform("cat", d, k, Sx, Sw)
    assert abs(O.alignment(O.apply_act_transform(X, Tk), O.apply_weight_transform(W, Tik)) /
               O.alignment(X @ T.T, W @ Ti) - 1) < 1e-10
    # an outlier channel is spread over all d channels by H_d, over its own block only by H_k
    ct_full = O.concentration_act(X @ T.T)
    ct_block = O.concentration_act(O.apply_act_transform(X, Tk))
    assert ct_full > ct_block


def test_full_rank_with_full_hadamard_reaches_the_ceiling():
    """k = d: M_hat is the full-rank optimum and H_d M_hat reaches A_max of Eq. 9 (R11)."""
    rng = _rng(71)
    d = 16
    X = rng.standard_normal((4000, d)) @ rng.standard_normal((d, d))
    W = rng.standard_normal((24, d))                 # d_out >= d: Sigma_w positive definite
    Sx = X.T @ X / X.shape[0]
    T, Ti, _, _ = O.build_transform_full_hadamard(d, d, Sx[None], (W.T @ W)[None])
    assert abs(O.alignment(X @ T.T, W @ Ti) / O.max_alignment(Sx, W) - 1) < 1e-8
    r = O.cat_layer_dense(X, W, T, Ti)
    assert np.isfinite(r["sqnr_db"]) and np.max(np.abs(r["qx"])) == 7
