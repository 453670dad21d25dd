"""Plain fp64 CPU oracle of the block Concentration-Alignment Transform (CAT) W4A4 linear layer.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg
of ``bench.py`` may import or run this module.  The CUDA library never calls it, and it shares
no code, table or constant with the CUDA path; both sides only take their inputs from the
seeded generators in ``workloads``.

Everything here follows the paper ("Dissecting Quantization Error: A Concentration-Alignment
Perspective") step by step, in float64, with numpy's LAPACK/BLAS routines (``eigh``,
``matmul``) as the only library primitives.  Conventions (Sec. 3, Eq. 5):

* a token is a row ``x`` of ``X`` [n, d_in]; the weight is ``W`` [d_out, d_in]; ``y = X W^T``.
* the transform ``T`` acts on activations online (``x' = T x``) and its inverse is folded
  into the weights offline (``W' = W T^{-1}``), so ``W' x' = W x``.
* block CAT (Sec. 4, Eq. 10) is block diagonal with ``d_in / k`` blocks of size ``k``;
  ``T_blocks[b]`` is the k x k block acting on channels ``b*k .. b*k+k-1``.

Readings where the paper is garbled or silent (listed with reasons in the design notes):

* INT4 grid: symmetric, step ``s = max|v| / 7``, codes in [-7, 7], round half to even.
  The paper's step ``r / (2^b - 1)`` with ``r = 2 max|v|`` has no zero level; the restricted
  symmetric grid keeps zero exact and never clips.  ``N_eff = r / s = 14`` is the number
  of intervals this grid has; ``N(b) = 2^b - 1`` is the paper's.
* Block CAT uses a k x k Sylvester Hadamard (orthonormal) in every block.
* Maximum alignment (Eq. 9) uses the eigenvalues ``mu_i`` of ``W Sigma_x W^T``:
  ``A_max = sum(mu) / (sum(sqrt(mu)))^2``.
* k = 1 (end of Sec. 4): ``m_i = (sum_j W_ji^2 / E[x_i^2]) ** (1/4)``.

Parity pins for every function live in ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional

import numpy as np

QMAX4 = 7  # largest INT4 code of the restricted symmetric grid


# ---------------------------------------------------------------------------------------------
# Quantizer: Lemma 2 (range r(x) = 2 max|x_i| for symmetric quantization), App. A.2.1 (uniform
# intervals of size s, round to nearest), Sec. 6 (activations per token, weights per output
# channel, round-to-nearest).
# ---------------------------------------------------------------------------------------------

RANGE_GRID = 100   # the L_2.4 search's candidate ranges are max|w| (RANGE_GRID - i) / RANGE_GRID


def quantize_rows_symmetric(V: np.ndarray, bits: int = 4, shrink: Optional[np.ndarray] = None):
    """Quantize every row of ``V`` on its own symmetric uniform grid.

    Returns ``(q, s, pre)``: integer codes (int64), the per-row step ``s = a / qmax`` and the
    pre-rounding values ``v / s = qmax * v / a`` (float64), where ``a = max|v|`` or, when the row's
    candidate index ``shrink[r] = i`` of the weight range search is given, the shrunk range
    ``a = max|v| (G - i) / G`` (G = RANGE_GRID).  An all-zero row gets ``s = 0`` and codes 0.

    The code is ``clamp(round_half_even(qmax * v / a), -qmax, qmax)``, evaluated in float64 as
    ``(G qmax v) / (max|v| (G - i))``.  For values with at most 24 significant bits (bf16 or fp32
    inputs, e.g. weights or activations under T = I) both operands are exact and the quotient is
    correctly rounded, so a real tie (a quotient of exactly m + 1/2) stays an exact tie and is broken
    to even, and every other quotient lies far beyond float64's rounding from a tie; the code is then
    the exact round-to-nearest of the definition."""
    V = np.asarray(V, dtype=np.float64)
    qmax = 2 ** (bits - 1) - 1
    amax = np.max(np.abs(V), axis=1) if V.shape[1] else np.zeros(V.shape[0])
    keep = np.full(V.shape[0], RANGE_GRID, dtype=np.float64) if shrink is None else \
        RANGE_GRID - np.asarray(shrink, dtype=np.float64)
    a = amax if shrink is None else amax * keep / RANGE_GRID
    s = a / qmax
    pre = np.zeros_like(V)
    nz = amax > 0
    pre[nz] = (RANGE_GRID * qmax * V[nz]) / (amax[nz] * keep[nz])[:, None]
    q = np.clip(np.rint(pre), -qmax, qmax).astype(np.int64)
    return q, s, pre


def quantize_rows_asymmetric(V: np.ndarray, bits: int = 4):
    """Per-row asymmetric uniform round-to-nearest quantizer (Sec. 6: activations are quantized
    dynamically per token, asymmetrically; Lemma 2: asymmetric range r = max - min, N(b) = 2^b - 1
    intervals).  Reading of the details the paper leaves open (the usual integer-zero-point grid):
    the range includes zero, ``lo = min(min v, 0)``, ``hi = max(max v, 0)``; the step is
    ``s = (hi - lo) / N``; the zero point is the integer ``z = round(-lo / s)``; the code is
    ``q = clamp(round(v / s) + z, 0, N)``, so ``Q(v) = s (q - z)`` and zero is exact.  Roundings are
    half to even; the quotients are evaluated in float64 as ``(N v) / (hi - lo)`` and
    ``(N (-lo)) / (hi - lo)``.  Returns ``(q, s, z, pre)`` with ``pre = N v / (hi - lo)``.  An
    all-zero row gets ``s = 0``, ``z = 0`` and codes 0."""
    V = np.asarray(V, dtype=np.float64)
    N = 2 ** bits - 1
    if V.shape[1]:
        lo = np.minimum(np.min(V, axis=1), 0.0)
        hi = np.maximum(np.max(V, axis=1), 0.0)
    else:
        lo = hi = np.zeros(V.shape[0])
    r = hi - lo
    s = r / N
    nz = r > 0
    pre = np.zeros_like(V)
    pre[nz] = (N * V[nz]) / r[nz, None]
    z = np.zeros(V.shape[0], dtype=np.int64)
    z[nz] = np.rint((N * -lo[nz]) / r[nz]).astype(np.int64)
    q = np.clip(np.rint(pre) + z[:, None], 0, N).astype(np.int64)
    q[~nz] = 0
    return q, s, z, pre


def dequantize_rows_asymmetric(q: np.ndarray, s: np.ndarray, z: np.ndarray) -> np.ndarray:
    """``Q(v) = s (q - z)`` per row."""
    return (q.astype(np.float64) - z[:, None]) * s[:, None]


def dequantize_rows(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    """``Q(v) = s * q`` per row."""
    return q.astype(np.float64) * s[:, None]


def weight_range_lp(W: np.ndarray, bits: int = 4, norm: float = 2.4, maxshrink: float = 0.8,
                    return_scores: bool = False):
    """Per-output-channel range search by the L_p error (Sec. 6: weight ranges are set with the
    L_2.4 norm, following GPTQ).  Candidates shrink the row's range, ``a_i = max|w| (G - i) / G``
    for ``i = 0 .. maxshrink * G - 1`` (G = RANGE_GRID); each is scored by
    ``sum_j |w_j - s_i q_ij|^norm`` with ``s_i = a_i / qmax`` and the codes of that range; the first
    candidate (the largest range) with the smallest score wins.  Returns the chosen candidate index
    per row (0 for an all-zero row), and with ``return_scores`` also every candidate's score
    [rows, candidates]."""
    W = np.asarray(W, dtype=np.float64)
    best = np.full(W.shape[0], np.inf)
    choice = np.zeros(W.shape[0], dtype=np.int64)
    scores = []
    for i in range(int(round(maxshrink * RANGE_GRID))):
        q, s, _ = quantize_rows_symmetric(W, bits, shrink=np.full(W.shape[0], i))
        err = np.sum(np.abs(W - q * s[:, None]) ** norm, axis=1)
        scores.append(err)
        better = err < best
        best[better] = err[better]
        choice[better] = i
    return (choice, np.stack(scores, axis=1)) if return_scores else choice


# ---------------------------------------------------------------------------------------------
# Matrix functions used by the alignment-optimal transform (Sec. 4, Eq. 7).
# ---------------------------------------------------------------------------------------------

def _sym(A: np.ndarray) -> np.ndarray:
    return 0.5 * (A + A.T)


def spd_power(A: np.ndarray, p: float) -> np.ndarray:
    """``A^p`` for a symmetric positive definite ``A``: ``V diag(lambda^p) V^T``."""
    lam, V = np.linalg.eigh(_sym(np.asarray(A, dtype=np.float64)))
    if lam[0] <= 0:
        raise np.linalg.LinAlgError("matrix is not positive definite")
    return _sym((V * lam ** p) @ V.T)


def geometric_mean(A: np.ndarray, B: np.ndarray) -> np.ndarray:
    """Matrix geometric mean (Sec. 4, Eq. 7): ``A # B = A^{1/2} (A^{-1/2} B A^{-1/2})^{1/2} A^{1/2}``."""
    Ah = spd_power(A, 0.5)
    Aih = spd_power(A, -0.5)
    return _sym(Ah @ spd_power(_sym(Aih @ B @ Aih), 0.5) @ Ah)


def alignment_optimal_M(Sigma_x: np.ndarray, Sigma_w: np.ndarray):
    """``M_hat = (Sigma_w # Sigma_x^{-1})^{1/2}`` (Sec. 4, Eq. 7).  Returns ``(M, M^{-1})``."""
    G = geometric_mean(Sigma_w, np.linalg.inv(Sigma_x))
    return spd_power(G, 0.5), spd_power(G, -0.5)


def hadamard(k: int) -> np.ndarray:
    """Orthonormal Sylvester Hadamard matrix of order k (a power of two): the +-1 matrix
    S_1 = [1], S_2m = [[S_m, S_m], [S_m, -S_m]], divided by sqrt(k)."""
    if k < 1 or k & (k - 1):
        raise ValueError("Hadamard order must be a power of two")
    S = np.ones((1, 1))
    while S.shape[0] < k:
        S = np.block([[S, S], [S, -S]])
    return S / np.sqrt(float(k))


# ---------------------------------------------------------------------------------------------
# Calibration statistics (Sec. 4: Sigma_x = E[x x^T], Sigma_w = W^T W; Eq. 10 keeps the k x k
# diagonal blocks).
# ---------------------------------------------------------------------------------------------

def calib_cov_block_sums(X: np.ndarray, k: int) -> np.ndarray:
    """Sums over tokens of ``x_b x_b^T`` for every diagonal k x k block: [d/k, k, k].  Dividing by
    the number of tokens gives the uncentered autocorrelation blocks of ``Sigma_x``."""
    X = np.asarray(X, dtype=np.float64)
    n, d = X.shape
    out = np.empty((d // k, k, k))
    for b in range(d // k):
        Xb = X[:, b * k:(b + 1) * k]
        out[b] = Xb.T @ Xb
    return out


def weight_autocorr_blocks(W: np.ndarray, k: int) -> np.ndarray:
    """Diagonal k x k blocks of ``Sigma_w = W^T W``: [d/k, k, k]."""
    W = np.asarray(W, dtype=np.float64)
    d_out, d = W.shape
    out = np.empty((d // k, k, k))
    for b in range(d // k):
        Wb = W[:, b * k:(b + 1) * k]
        out[b] = Wb.T @ Wb
    return out


# ---------------------------------------------------------------------------------------------
# Transforms (Sec. 3, Eq. 5; Sec. 4 two-step construction and Eq. 10).
# ---------------------------------------------------------------------------------------------

def build_transform(kind: str, d: int, k: int, Sigma_x_blocks: Optional[np.ndarray] = None,
                    Sigma_w_blocks: Optional[np.ndarray] = None, signs: Optional[np.ndarray] = None):
    """Block-diagonal transform ``T`` and its inverse, as [d/k, k, k] arrays.

    * ``identity``: T = I (plain RTN W4A4).
    * ``rht``: T_b = H_k Diag(sigma_b), sigma = the given random signs (a randomized Hadamard
      rotation; orthogonal, so it leaves alignment unchanged, Sec. 2 Eq. 4).
    * ``cat``: T_b = H_k M_hat_b with M_hat_b = (Sigma_w_b # Sigma_x_b^{-1})^{1/2} solved on the
      block's own k x k sub-problem (Sec. 4, Eq. 7 and Eq. 10)."""
    if d % k:
        raise ValueError("d must be a multiple of k")
    nb = d // k
    H = hadamard(k)
    T = np.empty((nb, k, k))
    Ti = np.empty((nb, k, k))
    for b in range(nb):
        if kind == "identity":
            T[b] = np.eye(k)
            Ti[b] = np.eye(k)
        elif kind == "rht":
            sg = np.asarray(signs, dtype=np.float64)[b * k:(b + 1) * k]
            T[b] = H * sg[None, :]
            Ti[b] = sg[:, None] * H.T
        elif kind == "cat":
            M, Mi = alignment_optimal_M(Sigma_x_blocks[b], Sigma_w_blocks[b])
            T[b] = H @ M
            Ti[b] = Mi @ H.T
        else:
            raise ValueError(kind)
    return T, Ti


def block_diag(blocks: np.ndarray) -> np.ndarray:
    """The dense d x d matrix of [d/k, k, k] diagonal blocks."""
    nb, k, _ = blocks.shape
    out = np.zeros((nb * k, nb * k))
    for b in range(nb):
        out[b * k:(b + 1) * k, b * k:(b + 1) * k] = blocks[b]
    return out


def build_transform_full_hadamard(d: int, k: int, Sigma_x_blocks: np.ndarray, Sigma_w_blocks: np.ndarray):
    """The approximately optimal transform of Sec. 4 with a full-size Hadamard: the block-diagonal
    alignment-optimal M_hat_block (Eq. 7 on every k x k block, Eq. 10) composed with the orthonormal
    Sylvester H_d over all d channels (d a power of two): T = H_d M_hat_block (dense d x d),
    T^{-1} = M_hat_block^{-1} H_d^T.  Returns ``(T, T^{-1}, M blocks, M^{-1} blocks)``."""
    nb = d // k
    M = np.empty((nb, k, k))
    Mi = np.empty((nb, k, k))
    for b in range(nb):
        M[b], Mi[b] = alignment_optimal_M(Sigma_x_blocks[b], Sigma_w_blocks[b])
    H = hadamard(d)
    return H @ block_diag(M), block_diag(Mi) @ H.T, M, Mi


def cat_layer_dense(X: np.ndarray, W: np.ndarray, T: np.ndarray, Tinv: np.ndarray) -> Dict[str, object]:
    """The layer with a dense transform (Sec. 3, Eq. 5): x' = T x, W' = W T^{-1}, per-token and
    per-channel symmetric INT4 codes, integer GEMM, SQNR against y = W x."""
    X = np.asarray(X, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    Xt = X @ T.T
    Wt = W @ Tinv
    qx, sx, pre_x = quantize_rows_symmetric(Xt)
    qw, sw, pre_w = quantize_rows_symmetric(Wt)
    acc, y_hat = w4a4_linear(qx, sx, qw, sw)
    y = linear(X, W)
    sig, err = sqnr_sums(y, y_hat)
    return dict(Xt=Xt, Wt=Wt, qx=qx, sx=sx, pre_x=pre_x, qw=qw, sw=sw, pre_w=pre_w, acc=acc, y_hat=y_hat, y=y,
                sqnr_db=10.0 * np.log10(sig / err))


def apply_act_transform(X: np.ndarray, T_blocks: np.ndarray) -> np.ndarray:
    """``x' = T x`` for every token row: ``X'_b = X_b T_b^T`` block by block."""
    X = np.asarray(X, dtype=np.float64)
    nb, k, _ = T_blocks.shape
    out = np.empty_like(X)
    for b in range(nb):
        out[:, b * k:(b + 1) * k] = X[:, b * k:(b + 1) * k] @ T_blocks[b].T
    return out


def apply_weight_transform(W: np.ndarray, Tinv_blocks: np.ndarray) -> np.ndarray:
    """``W' = W T^{-1}``: ``W'_b = W_b T_b^{-1}`` block by block."""
    W = np.asarray(W, dtype=np.float64)
    nb, k, _ = Tinv_blocks.shape
    out = np.empty_like(W)
    for b in range(nb):
        out[:, b * k:(b + 1) * k] = W[:, b * k:(b + 1) * k] @ Tinv_blocks[b]
    return out


# ---------------------------------------------------------------------------------------------
# Integer GEMM, dequantization and SQNR (Sec. 3 Eq. 5: y ~ Q(W T^{-1}) Q(T x); Sec. 2 Eq. 1).
# ---------------------------------------------------------------------------------------------

def int_gemm(qx: np.ndarray, qw: np.ndarray) -> np.ndarray:
    """``acc[t, o] = sum_i qx[t, i] qw[o, i]`` exactly.  The products and every partial sum are
    integers far below 2^53, so a float64 matmul is exact; the result is returned as int64."""
    acc = np.asarray(qx, dtype=np.float64) @ np.asarray(qw, dtype=np.float64).T
    return np.rint(acc).astype(np.int64)


def dequantize_output(acc: np.ndarray, sx: np.ndarray, sw: np.ndarray) -> np.ndarray:
    """``y_hat[t, o] = acc[t, o] * s_x[t] * s_w[o]``."""
    return acc.astype(np.float64) * sx[:, None] * sw[None, :]


def linear(X: np.ndarray, W: np.ndarray) -> np.ndarray:
    """Full-precision layer output ``y = W x`` for every token."""
    return np.asarray(X, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T


def sqnr_sums(y: np.ndarray, y_hat: np.ndarray):
    """``(sum y^2, sum (y - y_hat)^2)`` over all tokens and outputs."""
    y = np.asarray(y, dtype=np.float64)
    e = y - np.asarray(y_hat, dtype=np.float64)
    return float(np.sum(y * y)), float(np.sum(e * e))


def sqnr_db(y: np.ndarray, y_hat: np.ndarray) -> float:
    """SQNR (Sec. 2, Eq. 1) in dB: ``10 log10(E||W x||^2 / E||W x - W~ x~||^2)``."""
    sig, err = sqnr_sums(y, y_hat)
    return 10.0 * np.log10(sig / err)


# ---------------------------------------------------------------------------------------------
# The whole layer.
# ---------------------------------------------------------------------------------------------

@dataclasses.dataclass
class PreparedWeights:
    T: np.ndarray          # [d/k, k, k] activation transform blocks
    Tinv: np.ndarray       # [d/k, k, k]
    Wt: np.ndarray         # W T^{-1}
    qw: np.ndarray         # int64 codes [d_out, d_in]
    sw: np.ndarray         # per-output-channel steps [d_out]
    pre_w: np.ndarray      # pre-rounding values
    shrink: Optional[np.ndarray] = None  # per-row candidate index of the L_p range search (None: max range)


def prepare_weights(W: np.ndarray, kind: str, k: int, X_calib: Optional[np.ndarray] = None,
                    signs: Optional[np.ndarray] = None, Sigma_x_blocks: Optional[np.ndarray] = None,
                    bits: int = 4, w_range: str = "max") -> PreparedWeights:
    """Offline part: calibration statistics, transform, ``W T^{-1}`` and its per-channel b-bit
    symmetric codes; ``w_range`` = "max" (the row maximum) or "l2.4" (the L_2.4 range search, Sec. 6)."""
    W = np.asarray(W, dtype=np.float64)
    d = W.shape[1]
    Sx = Sw = None
    if kind == "cat":
        if Sigma_x_blocks is None:
            Xc = np.asarray(X_calib, dtype=np.float64)
            Sigma_x_blocks = calib_cov_block_sums(Xc, k) / Xc.shape[0]
        Sx = Sigma_x_blocks
        Sw = weight_autocorr_blocks(W, k)
    T, Ti = build_transform(kind, d, k, Sx, Sw, signs)
    Wt = apply_weight_transform(W, Ti)
    shrink = weight_range_lp(Wt, bits) if w_range == "l2.4" else None
    qw, sw, pre_w = quantize_rows_symmetric(Wt, bits, shrink=shrink)
    return PreparedWeights(T=T, Tinv=Ti, Wt=Wt, qw=qw, sw=sw, pre_w=pre_w, shrink=shrink)


@dataclasses.dataclass
class ActCodes:
    Xt: np.ndarray        # T x for every token
    qx: np.ndarray        # int64 codes [n, d_in]
    sx: np.ndarray        # per-token steps [n]
    pre_x: np.ndarray
    zx: Optional[np.ndarray] = None   # per-token zero points (asymmetric), else None


def transform_quantize_act(X: np.ndarray, T_blocks: np.ndarray, bits: int = 4,
                           asymmetric: bool = False) -> ActCodes:
    """Online part, first half: ``x' = T x`` and its per-token b-bit codes (symmetric, or the
    asymmetric per-token quantizer of Sec. 6)."""
    Xt = apply_act_transform(X, T_blocks)
    if asymmetric:
        qx, sx, zx, pre = quantize_rows_asymmetric(Xt, bits)
        return ActCodes(Xt=Xt, qx=qx, sx=sx, pre_x=pre, zx=zx)
    qx, sx, pre = quantize_rows_symmetric(Xt, bits)
    return ActCodes(Xt=Xt, qx=qx, sx=sx, pre_x=pre)


def w4a4_linear(qx, sx, qw, sw, zx=None):
    """Online part, second half: integer GEMM and dequantization.  Returns ``(acc, y_hat)`` with
    ``acc[t, o] = sum_i (qx[t, i] - zx[t]) qw[o, i]`` (``zx`` = 0 for symmetric activations); the name
    stays from the 4-bit layer, the arithmetic holds for every bit width."""
    qx = np.asarray(qx, dtype=np.int64)
    if zx is not None:
        qx = qx - np.asarray(zx, dtype=np.int64)[:, None]
    acc = int_gemm(qx, qw)
    return acc, dequantize_output(acc, sx, sw)


def cat_layer(X: np.ndarray, W: np.ndarray, kind: str, k: int, X_calib: Optional[np.ndarray] = None,
              signs: Optional[np.ndarray] = None, bits_x: int = 4, bits_w: int = 4, act_asym: bool = False,
              w_range: str = "max") -> Dict[str, object]:
    """Every step of the layer, in the paper's order, returning all intermediates (W{bits_w}A{bits_x};
    Sec. 6's set-up is ``act_asym=True, w_range="l2.4"``)."""
    pw = prepare_weights(W, kind, k, X_calib=X_calib, signs=signs, bits=bits_w, w_range=w_range)
    ac = transform_quantize_act(X, pw.T, bits=bits_x, asymmetric=act_asym)
    acc, y_hat = w4a4_linear(ac.qx, ac.sx, pw.qw, pw.sw, zx=ac.zx)
    y = linear(X, W)
    sig, err = sqnr_sums(y, y_hat)
    return dict(prep=pw, act=ac, acc=acc, y_hat=y_hat, y=y, sig=sig, err=err,
                sqnr_db=10.0 * np.log10(sig / err))


# ---------------------------------------------------------------------------------------------
# Analysis quantities (Sec. 2: Lemma 1-3, Theorem 1, concentration and alignment; Sec. 4 Eq. 9).
# ---------------------------------------------------------------------------------------------

def parallel(a: float, b: float) -> float:
    """``a || b = (1/a + 1/b)^{-1}`` (Lemma 1)."""
    return 1.0 / (1.0 / a + 1.0 / b)


def range_symmetric(V: np.ndarray) -> np.ndarray:
    """``r(v) = 2 max_i |v_i|`` per row (Lemma 2)."""
    return 2.0 * np.max(np.abs(np.asarray(V, dtype=np.float64)), axis=1)


def range_asymmetric(V: np.ndarray) -> np.ndarray:
    """``r(v) = max_i v_i - min_i v_i`` per row (Lemma 2)."""
    V = np.asarray(V, dtype=np.float64)
    return np.max(V, axis=1) - np.min(V, axis=1)


def concentration_act(X: np.ndarray, symmetric: bool = True) -> float:
    """``C(x) = E||x||^2 / E[r(x)^2]`` over tokens (Lemma 2)."""
    X = np.asarray(X, dtype=np.float64)
    r = range_symmetric(X) if symmetric else range_asymmetric(X)
    return float(np.mean(np.sum(X * X, axis=1)) / np.mean(r * r))


def concentration_weight(W: np.ndarray) -> float:
    """``C(W) = sum_i ||w_i||^2 / sum_i r(w_i)^2`` over output rows (Lemma 3)."""
    W = np.asarray(W, dtype=np.float64)
    r = range_symmetric(W)
    return float(np.sum(W * W) / np.sum(r * r))


def alignment(X: np.ndarray, W: np.ndarray) -> float:
    """``A(x, W) = E||W x||^2 / (||W||_F^2 E||x||^2)`` (Lemma 2)."""
    X = np.asarray(X, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    Y = X @ W.T
    return float(np.mean(np.sum(Y * Y, axis=1)) / (np.sum(W * W) * np.mean(np.sum(X * X, axis=1))))


def alignment_from_moments(Sigma_x: np.ndarray, Sigma_w: np.ndarray) -> float:
    """``A = Tr(Sigma_w Sigma_x) / (Tr(Sigma_w) Tr(Sigma_x))``: the same ratio written with
    ``E||W x||^2 = Tr(W^T W E[x x^T])``."""
    return float(np.trace(Sigma_w @ Sigma_x) / (np.trace(Sigma_w) * np.trace(Sigma_x)))


def max_alignment(Sigma_x: np.ndarray, W: np.ndarray) -> float:
    """Largest alignment reachable by an invertible transform (Sec. 4, Eq. 9), in terms of the
    eigenvalues ``mu_i`` of ``Sigma_y = W Sigma_x W^T``: ``sum(mu) / (sum(sqrt(mu)))^2``."""
    W = np.asarray(W, dtype=np.float64)
    mu = np.linalg.eigvalsh(_sym(W @ Sigma_x @ W.T))
    mu = np.clip(mu, 0.0, None)
    return float(np.sum(mu) / np.sum(np.sqrt(mu)) ** 2)


def sqnr_act_only(X: np.ndarray, W: np.ndarray, bits: int = 4) -> float:
    """Measured ``SQNR(W x~)``: only activations quantized (per token)."""
    q, s, _ = quantize_rows_symmetric(X, bits)
    return 10 ** (sqnr_db(linear(X, W), linear(dequantize_rows(q, s), W)) / 10)


def sqnr_weight_only(X: np.ndarray, W: np.ndarray, bits: int = 4) -> float:
    """Measured ``SQNR(W~ x)``: only weights quantized (per output channel)."""
    q, s, _ = quantize_rows_symmetric(W, bits)
    return 10 ** (sqnr_db(linear(X, W), linear(X, dequantize_rows(q, s))) / 10)


def sqnr_both(X: np.ndarray, W: np.ndarray, bits_x: int = 4, bits_w: int = 4) -> float:
    """Measured ``SQNR(W~ x~)`` (Sec. 2, Eq. 1), linear scale."""
    qx, sx, _ = quantize_rows_symmetric(X, bits_x)
    qw, sw, _ = quantize_rows_symmetric(W, bits_w)
    return 10 ** (sqnr_db(linear(X, W), linear(dequantize_rows(qx, sx), dequantize_rows(qw, sw))) / 10)


def n_intervals(bits: int, paper: bool = False) -> float:
    """Number of quantization intervals across the range: the paper's ``N(b) = 2^b - 1``, or the
    ``2 (2^{b-1} - 1)`` intervals of the restricted symmetric grid used here (``r / s``)."""
    return float(2 ** bits - 1) if paper else float(2 * (2 ** (bits - 1) - 1))


def lemma2_act_sqnr(X: np.ndarray, W: np.ndarray, bits: int = 4, paper_N: bool = False) -> float:
    """Lemma 2: ``SQNR(W x~) ~ 12 N(b_x)^2 C(x) A(x, W)``."""
    return 12.0 * n_intervals(bits, paper_N) ** 2 * concentration_act(X) * alignment(X, W)


def lemma3_weight_sqnr(X: np.ndarray, W: np.ndarray, bits: int = 4, paper_N: bool = False) -> float:
    """Lemma 3: ``SQNR(W~ x) ~ 12 N(b_w)^2 C(W) A(x, W)``."""
    return 12.0 * n_intervals(bits, paper_N) ** 2 * concentration_weight(W) * alignment(X, W)


def theorem1_sqnr(X: np.ndarray, W: np.ndarray, bits_x: int = 4, bits_w: int = 4, paper_N: bool = False) -> float:
    """Theorem 1: ``SQNR ~ 12 (N(b_x)^2 C(x) || N(b_w)^2 C(W)) A(x, W)``."""
    nx, nw = n_intervals(bits_x, paper_N), n_intervals(bits_w, paper_N)
    return 12.0 * parallel(nx ** 2 * concentration_act(X), nw ** 2 * concentration_weight(W)) * alignment(X, W)


def db(v: float) -> float:
    return 10.0 * np.log10(v)
