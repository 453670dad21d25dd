"""The C-ABI library without a GPU: it builds, loads, exports every entry point declared in
include/cat_w4a4.h, validates arguments on the host before any CUDA call, and its host-side
float64 transform construction matches the oracle."""
import ctypes
import os

import numpy as np
import pytest

import oracle as O
import paper_2603_04359_gb300 as cat
from paper_2603_04359_gb300 import build as catbuild

CSRC = os.path.join(os.path.dirname(catbuild.__file__), "csrc")


@pytest.fixture(scope="session")
def lib():
    srcs = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    stale = (not os.path.exists(cat.library_path()) or
             max(os.path.getmtime(s) for s in srcs) > os.path.getmtime(cat.library_path()))
    if stale:
        catbuild.build()
    return cat.load_library()


def test_exports_every_declared_symbol(lib):
    names = cat.exported_symbols()
    for expected in ("cat_calib_cov", "cat_quantize_weights", "cat_transform_quantize_act", "cat_w4a4_linear",
                     "cat_sqnr", "cat_status_string", "cat_build_transform_host", "cat_device_status"):
        assert expected in names
    for name in names:
        assert hasattr(lib, name), name


def test_status_strings_and_version(lib):
    assert lib.cat_status_string(0) == b"CAT_OK"
    assert lib.cat_status_string(7) == b"CAT_ERR_TIMEOUT"
    assert cat.cat_version() >= 10000


def _fake(addr):
    return ctypes.c_void_p(addr)


def test_host_validation_without_gpu(lib):
    """Invalid calls are rejected before anything touches CUDA (so this runs on a CPU machine)."""
    P = _fake(0x10000)
    bad = _fake(0x10008)  # not 16-byte aligned
    # cat_transform_quantize_act(x, dtype, n, d_in, k, T, xq, sx, stream)
    assert lib.cat_transform_quantize_act(P, 1, 4, 48, 16, P, P, P, None) == 2          # d_in % 32
    assert lib.cat_transform_quantize_act(P, 1, 4, 64, 48, P, P, P, None) == 2          # k not a power of two
    assert lib.cat_transform_quantize_act(P, 1, 4, 96, 64, P, P, P, None) == 2          # k does not divide d_in
    assert lib.cat_transform_quantize_act(P, 7, 4, 64, 32, P, P, P, None) == 1          # dtype
    assert lib.cat_transform_quantize_act(None, 1, 4, 64, 32, P, P, P, None) == 1       # NULL
    assert lib.cat_transform_quantize_act(bad, 1, 4, 64, 32, P, P, P, None) == 3        # alignment
    assert lib.cat_transform_quantize_act(P, 1, -1, 64, 32, P, P, P, None) == 2         # n < 0
    assert lib.cat_transform_quantize_act(P, 1, 0, 64, 32, None, None, None, None) == 0  # n == 0: no-op
    lib.cat_transform_quantize_act(P, 1, 4, 48, 16, P, P, P, None)
    assert b"multiple of 32" in lib.cat_last_error()
    # cat_w4a4_linear(xq, sx, wq, sw, n, d_in, d_out, y, acc, stream)
    assert lib.cat_w4a4_linear(P, P, P, P, 4, 300000, 8, P, None, None) == 2            # exactness bound
    assert lib.cat_w4a4_linear(P, P, P, P, 4, 64, 0, P, None, None) == 2                # d_out
    assert lib.cat_w4a4_linear(P, P, P, P, 4, 64, 8, None, None, None) == 1             # y NULL
    assert lib.cat_w4a4_linear(P, P, P, P, 4, 64, 8, P, bad, None) == 3                 # acc alignment
    # cat_calib_cov(x, dtype, n, d, k, sigma, accumulate, stream)
    assert lib.cat_calib_cov(P, 0, 4, 100, 32, P, 0, None) == 2
    assert lib.cat_calib_cov(P, 0, 4, 64, 32, None, 0, None) == 1
    # cat_quantize_weights(W, dtype, d_out, d_in, k, kind, sigma_x, n_calib, signs, T, Wq, sw, stream)
    assert lib.cat_quantize_weights(P, 1, 8, 64, 32, 2, None, 0, None, P, P, P, None) == 1   # CAT w/o sigma
    assert lib.cat_quantize_weights(P, 1, 8, 64, 32, 1, None, 0, None, P, P, P, None) == 1   # RHT w/o signs
    assert lib.cat_quantize_weights(P, 1, 8, 64, 32, 9, None, 0, None, P, P, P, None) == 1   # kind
    # cat_sqnr(y_ref, y_hat, numel, out3, stream)
    assert lib.cat_sqnr(P, P, -1, P, None) == 2
    assert lib.cat_sqnr(P, None, 10, P, None) == 1
    # byte codes: cat_codes_to_e4m3(codes, rows, d, out, stream)
    assert lib.cat_codes_to_e4m3(P, 4, 48, P, None) == 2                                 # d % 32
    assert lib.cat_codes_to_e4m3(P, -1, 64, P, None) == 2                                # rows < 0
    assert lib.cat_codes_to_e4m3(P, 0, 64, None, None) == 0                              # rows == 0: no-op
    assert lib.cat_codes_to_e4m3(P, 4, 64, None, None) == 1                              # NULL
    assert lib.cat_codes_to_e4m3(bad, 4, 64, P, None) == 3                               # alignment
    # cat_transform_quantize_act_e8(x, dtype, n, d_in, k, T, T_planes, xq8, sx, stream)
    assert lib.cat_transform_quantize_act_e8(P, 1, 4, 48, 16, P, None, P, P, None) == 2  # d_in % 32
    assert lib.cat_transform_quantize_act_e8(P, 7, 4, 64, 32, P, None, P, P, None) == 1  # dtype
    assert lib.cat_transform_quantize_act_e8(P, 1, 4, 64, 32, P, None, None, P, None) == 1   # NULL xq8
    assert lib.cat_transform_quantize_act_e8(P, 1, 4, 64, 32, P, bad, P, P, None) == 3   # planes alignment
    assert lib.cat_transform_quantize_act_e8(P, 1, 0, 64, 32, None, None, None, None, None) == 0
    # cat_w4a4_linear_e8(xq8, sx, wq8, sw, n, d_in, d_out, y, acc, stream) and the SQNR variant
    assert lib.cat_w4a4_linear_e8(P, P, P, P, 4, 300000, 8, P, None, None) == 2         # exactness bound
    assert lib.cat_w4a4_linear_e8(P, P, P, P, 4, 64, 0, P, None, None) == 2             # d_out
    assert lib.cat_w4a4_linear_e8(P, P, P, P, 4, 64, 8, None, None, None) == 1          # y NULL
    assert lib.cat_w4a4_linear_e8(P, P, bad, P, 4, 64, 8, P, None, None) == 3           # alignment
    assert lib.cat_w4a4_linear_sqnr_e8(P, P, P, P, 4, 64, 8, P, P, None, None) == 1     # out3 NULL
    assert lib.cat_w4a4_linear_sqnr_e8(P, P, P, P, 4, 96, 8, P, bad, P, None) == 3      # y_ref alignment


def test_valid_call_without_device_reports_cuda_error(lib):
    try:
        import torch
        if torch.cuda.is_available():
            pytest.skip("a GPU is present")
    except ImportError:
        pass
    P = _fake(0x10000)
    st = lib.cat_transform_quantize_act(P, 1, 4, 64, 32, P, P, P, None)
    assert st in (5, 6)
    assert len(lib.cat_last_error()) > 0


def _blocks_problem(seed, d, k, n=800):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, d)) @ (rng.standard_normal((d, d)) / np.sqrt(d) + np.eye(d))
    X[:, rng.choice(d, 2, replace=False)] *= 60.0
    W = rng.standard_normal((3 * d // 2, d)) * 0.02 * rng.lognormal(0, 0.5, (3 * d // 2, 1))
    return X, W, rng.choice([-1.0, 1.0], d)


@pytest.mark.parametrize("k", [16, 32, 64])
def test_host_transform_matches_oracle(lib, k):
    d = 128
    X, W, signs = _blocks_problem(k, d, k)
    Sx_sum = O.calib_cov_block_sums(X, k)
    Sw = O.weight_autocorr_blocks(W, k)
    for kind in ("identity", "rht", "cat"):
        T, Ti = cat.cat_build_transform_host(kind, d, k, Sx_sum, X.shape[0], Sw, signs)
        To, Tio = O.build_transform(kind, d, k, Sx_sum / X.shape[0], Sw, signs)
        rel = np.linalg.norm(T - To) / np.linalg.norm(To)
        reli = np.linalg.norm(Ti - Tio) / np.linalg.norm(Tio)
        assert rel < 1e-9 and reli < 1e-9, (kind, rel, reli)
        for b in range(d // k):
            np.testing.assert_allclose(T[b] @ Ti[b], np.eye(k), atol=1e-9)


def test_host_transform_k256_and_errors(lib):
    d, k = 256, 256
    X, W, signs = _blocks_problem(7, d, k, n=1500)
    Sx_sum = O.calib_cov_block_sums(X, k)
    Sw = O.weight_autocorr_blocks(W, k)
    T, Ti = cat.cat_build_transform_host("cat", d, k, Sx_sum, X.shape[0], Sw)
    To, Tio = O.build_transform("cat", d, k, Sx_sum / X.shape[0], Sw)
    assert np.linalg.norm(T - To) / np.linalg.norm(To) < 1e-8
    # a singular calibration block is rejected
    Sx_bad = Sx_sum.copy()
    Sx_bad[0] = 0.0
    with pytest.raises(cat.CatError) as ei:
        cat.cat_build_transform_host("cat", d, k, Sx_bad, X.shape[0], Sw)
    assert ei.value.status == 4
    with pytest.raises(cat.CatError):
        cat.cat_build_transform_host("rht", d, k, rht_signs=np.full(d, 0.5))


def test_wait_limit_setter_rejects_bounds_above_one_second():
    """The testing aid refuses a bound above the default before any CUDA call (runs without a GPU)."""
    import ctypes
    lib = cat.load_library()
    assert lib.cat_set_wait_limit_ns(ctypes.c_uint64(2_000_000_000)) == 1      # CAT_ERR_INVALID_ARG
    assert b"at most 1 s" in lib.cat_last_error()


def test_host_builder_diagonal_and_full_hadamard_kinds_match_the_oracle():
    """kind 3 (k = 1 optimum in k-blocks) and kind 4 (the M_b blocks of CAT with the full-size
    Hadamard) against the oracle (host only)."""
    rng = np.random.default_rng(81)
    d, k = 64, 16
    X = rng.standard_normal((500, d)) @ (rng.standard_normal((d, d)) * 0.3 + np.eye(d))
    W = rng.standard_normal((80, d)) * 0.05
    sx = O.calib_cov_block_sums(X, k)
    sw = O.weight_autocorr_blocks(W, k)
    T3, Ti3 = cat.cat_build_transform_host("cat_diag", d, k, sigma_x=sx, n_calib=X.shape[0], sigma_w=sw)
    m = (np.sum(W * W, axis=0) / np.mean(X * X, axis=0)) ** 0.25          # end of Sec. 4 (R9)
    np.testing.assert_allclose(O.block_diag(T3), np.diag(m), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(O.block_diag(Ti3), np.diag(1 / m), rtol=1e-12, atol=1e-15)
    Tk1, _ = O.build_transform("cat", d, 1, O.calib_cov_block_sums(X, 1) / X.shape[0], O.weight_autocorr_blocks(W, 1))
    np.testing.assert_allclose(np.diag(O.block_diag(T3)), Tk1[:, 0, 0], rtol=1e-10)
    T4, Ti4 = cat.cat_build_transform_host("cat_hd", d, k, sigma_x=sx, n_calib=X.shape[0], sigma_w=sw)
    _, _, M, Mi = O.build_transform_full_hadamard(d, k, sx / X.shape[0], sw)
    np.testing.assert_allclose(T4, M, rtol=1e-8, atol=1e-10)
    np.testing.assert_allclose(Ti4, Mi, rtol=1e-8, atol=1e-10)


def test_alignment_ceiling_host_matches_eq9():
    rng = np.random.default_rng(82)
    d = 48
    X = rng.standard_normal((3000, d)) @ rng.standard_normal((d, d))
    W = rng.standard_normal((30, d))                       # rank-deficient Sigma_w is allowed
    Sx = X.T @ X / X.shape[0]
    a, s_mu, s_sq = cat.cat_alignment_ceiling_host(Sx, W.T @ W)
    # P = Sx^1/2 Sw Sx^1/2 is 48 x 48 of rank 30: its 18 zero eigenvalues come out of the float64
    # eigen-decomposition at ~1e-14 of the largest, whose square roots add ~1e-8 to sum sqrt(mu)
    assert abs(a / O.max_alignment(Sx, W) - 1) < 1e-7
    mu = np.clip(np.linalg.eigvalsh(W @ Sx @ W.T), 0, None)
    assert abs(s_mu / mu.sum() - 1) < 1e-9 and abs(s_sq / np.sqrt(mu).sum() - 1) < 1e-7
    with pytest.raises(cat.CatError):
        cat.cat_alignment_ceiling_host(-np.eye(4), np.eye(4))
