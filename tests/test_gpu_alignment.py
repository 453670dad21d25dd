"""The alignment ceiling, the k = 1 diagonal optimum and the full-size Hadamard (Sec. 4) through the
library, against the oracle.  Tolerances as test_gpu_parity.py: codes +-1 at rounding boundaries,
y 1e-3 relative Frobenius, SQNR 0.01 dB; the ceiling from GPU statistics within 0.01 dB."""
import numpy as np
import pytest
import torch

import oracle as O
import sm4x8
import workloads as WL
from test_gpu_parity import DEV, check_codes, rel_fro, to_dev

pytestmark = pytest.mark.gpu

cat = pytest.importorskip("paper_2603_04359_gb300")


@pytest.mark.parametrize("rows,d", [(1, 2), (7, 64), (300, 1024), (33, 8192), (3, 32768)])
def test_fwht_rows(rows, d):
    rng = np.random.default_rng(rows + d)
    V = rng.standard_normal((rows, d)).astype(np.float32)
    out = cat.cat_fwht_rows(torch.from_numpy(V).to(DEV)).cpu().numpy()
    if d <= 8192:
        ref = V.astype(np.float64) @ O.hadamard(d).T
    else:                                                   # H_2d = [[H, H], [H, -H]] / sqrt(2)
        Hh = O.hadamard(d // 2)
        a, b = V[:, : d // 2].astype(np.float64) @ Hh.T, V[:, d // 2:].astype(np.float64) @ Hh.T
        ref = np.hstack([a + b, a - b]) / np.sqrt(2.0)
    assert rel_fro(out, ref) < 1e-6


@pytest.mark.parametrize("n,d,dtype", [(1, 1, "f32"), (300, 200, "bf16"), (1000, 512, "f32")])
def test_gram(n, d, dtype):
    rng = np.random.default_rng(n + d)
    X = WL.cast(rng.standard_normal((n, d)) * rng.lognormal(0, 1, d), dtype)
    C = cat.cat_gram_f32(to_dev(X)).cpu().numpy()
    assert rel_fro(C, X.values.T @ X.values) < 1e-6


LAYER = WL.small_config("align", d_in=512, d_out=768, n_eval=300, n_calib=1024, k=64, seed=91)


@pytest.mark.parametrize("k", [16, 64])
def test_diagonal_cat_layer(k):
    """kind "cat_diag": the k = 1 optimum m_i = (sum_j W_ji^2 / E[x_i^2])^{1/4} (end of Sec. 4), stored in k-blocks."""
    L = WL.make_layer(LAYER)
    x, W, xc = to_dev(L.x_eval), to_dev(L.W), to_dev(L.x_calib)
    sig = cat.cat_calib_cov(xc, k)
    T, Wq, sw = cat.cat_quantize_weights(W, k, "cat_diag", sigma_x=sig, n_calib=LAYER.n_calib)
    xq, sx = cat.cat_transform_quantize_act(x, T, k)
    y = cat.cat_w4a4_linear(xq, sx, Wq, sw).cpu().numpy()
    ref = O.cat_layer(L.x_eval.values, L.W.values, "cat", 1, X_calib=L.x_calib.values)
    np.testing.assert_allclose(np.diagonal(O.block_diag(T.double().cpu().numpy())), ref["prep"].T[:, 0, 0], rtol=1e-5)
    check_codes(sm4x8.unpack(Wq.cpu().numpy()), ref["prep"].qw, ref["prep"].pre_w)
    check_codes(sm4x8.unpack(xq.cpu().numpy()), ref["act"].qx, ref["act"].pre_x)
    assert rel_fro(y, ref["y_hat"]) < 1e-3
    s3 = cat.cat_sqnr(torch.from_numpy(ref["y"].astype(np.float32)).to(DEV), torch.from_numpy(y).to(DEV)).cpu().numpy()
    assert abs(s3[2] - ref["sqnr_db"]) < 0.01
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("k", [16, 64])
def test_full_hadamard_cat_layer(k):
    """kind "cat_hd": T = H_d M_block (Sec. 4) -- the block optimum with the Hadamard over all channels."""
    L = WL.make_layer(LAYER)
    x, W, xc = to_dev(L.x_eval), to_dev(L.W), to_dev(L.x_calib)
    sig = cat.cat_calib_cov(xc, k)
    M, Wq, sw = cat.cat_quantize_weights(W, k, "cat_hd", sigma_x=sig, n_calib=LAYER.n_calib)
    xq, sx = cat.cat_transform_quantize_act_hd(x, M, k)
    y = cat.cat_w4a4_linear(xq, sx, Wq, sw).cpu().numpy()
    Sx = O.calib_cov_block_sums(L.x_calib.values, k) / LAYER.n_calib
    T, Ti, Mo, _ = O.build_transform_full_hadamard(LAYER.d_in, k, Sx, O.weight_autocorr_blocks(L.W.values, k))
    assert rel_fro(M.cpu().numpy(), Mo) < 1e-5
    ref = O.cat_layer_dense(L.x_eval.values, L.W.values, T, Ti)
    check_codes(sm4x8.unpack(Wq.cpu().numpy()), ref["qw"], ref["pre_w"])
    check_codes(sm4x8.unpack(xq.cpu().numpy()), ref["qx"], ref["pre_x"])
    np.testing.assert_allclose(sx.cpu().numpy(), ref["sx"], rtol=1e-5)
    assert rel_fro(y, ref["y_hat"]) < 1e-3
    s3 = cat.cat_sqnr(torch.from_numpy(ref["y"].astype(np.float32)).to(DEV), torch.from_numpy(y).to(DEV)).cpu().numpy()
    assert abs(s3[2] - ref["sqnr_db"]) < 0.01
    assert cat.cat_device_status()[0] == 0


def test_alignment_ceiling_from_gpu_statistics():
    """A_max (Eq. 9) from the full Sigma_x and Sigma_w formed on the GPU, against the oracle's; the block
    CAT alignments stay below it and grow with k (Sec. 4: larger blocks approach the full-rank optimum)."""
    L = WL.make_layer(LAYER)
    xc, W = to_dev(L.x_calib), to_dev(L.W)
    Sx = cat.cat_gram_f32(xc).double().cpu().numpy() / LAYER.n_calib
    Sw = cat.cat_gram_f32(W).double().cpu().numpy()
    a_max, _, _ = cat.cat_alignment_ceiling_host(Sx, Sw)
    Sx_ref = L.x_calib.values.T.astype(np.float64) @ L.x_calib.values / LAYER.n_calib
    a_ref = O.max_alignment(Sx_ref, L.W.values)
    assert abs(10 * np.log10(a_max / a_ref)) < 0.01
    prev = 0.0
    for k in (16, 64, 256):
        T, Ti = O.build_transform("cat", LAYER.d_in, k, O.calib_cov_block_sums(L.x_calib.values, k) / LAYER.n_calib,
                                  O.weight_autocorr_blocks(L.W.values, k))
        Tb, Tib = O.block_diag(T), O.block_diag(Ti)         # x' = T x: Sigma_x' = T Sigma_x T^T; W' = W T^-1
        a_k = O.alignment_from_moments(Tb @ Sx_ref @ Tb.T, Tib.T @ L.W.values.T @ L.W.values @ Tib)
        assert a_k <= a_max * (1 + 1e-6) and a_k >= prev * (1 - 1e-6)
        prev = a_k
