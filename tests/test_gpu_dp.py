"""Bit widths and Sec. 6's quantizer set-up through the digit-plane path, against the oracle.

Tolerances as the W4A4 parity tests: accumulators bit-exact given identical codes; codes within +-1
only where the oracle's pre-rounding value lies within 1e-5 (relative) of a rounding boundary, in at
most 1e-4 of the elements (at least one); exact codes under T = I (the quantizer sees the inputs);
steps 1e-5 relative; y 1e-3 relative Frobenius; SQNR 0.01 dB.  The L_2.4 range may pick another
candidate than the oracle only where the oracle's scores of the two candidates agree to 1e-5."""
import numpy as np
import pytest
import torch

import dp_planes
import oracle as O
import workloads as WL

pytestmark = pytest.mark.gpu

cat = pytest.importorskip("paper_2603_04359_gb300")
DEV = "cuda"


def to_dev(t: WL.Tensor) -> torch.Tensor:
    if t.dtype == "f32":
        return torch.from_numpy(np.ascontiguousarray(t.raw)).to(DEV)
    return torch.from_numpy(np.ascontiguousarray(t.raw).view(np.int16)).view(torch.bfloat16).to(DEV)


def check_codes(q_gpu, q_ref, pre_ref, rel=1e-5, frac=1e-4):
    diff = np.asarray(q_gpu) - q_ref
    bad = diff != 0
    if not bad.any():
        return 0
    assert np.abs(diff).max() <= 1, "codes differ by more than 1"
    a = np.abs(pre_ref[bad])
    boundary = np.floor(a) + 0.5
    assert np.all(np.abs(a - boundary) <= rel * boundary), "a code differs away from a rounding boundary"
    assert bad.sum() <= max(1, frac * q_ref.size), f"{bad.sum()} codes differ (> {frac} of {q_ref.size})"
    return int(bad.sum())


def rel_fro(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-300))


def test_dp_planes_count():
    assert [cat.cat_dp_planes(b) for b in (1, 2, 3, 4, 5, 6, 8, 9)] == [0, 1, 1, 1, 2, 2, 2, 0]


# ------------------------------------------------------------------------------------------
# cat_linear_dp: exact accumulators given identical codes
# ------------------------------------------------------------------------------------------

def _rand_codes(rng, shape, bits, asym):
    if asym:
        return rng.integers(0, 2 ** bits, shape)
    qm = 2 ** (bits - 1) - 1
    return rng.integers(-qm, qm + 1, shape)


DP_GEMM = [  # (n, d_in, d_out, bits_x, bits_w, asym_x)
    (130, 256, 200, 8, 8, False), (64, 1024, 128, 6, 6, False), (300, 544, 333, 8, 4, False),
    (128, 128, 128, 4, 8, False), (257, 2048, 520, 4, 4, False), (5, 96, 17, 3, 5, False),
    (200, 384, 256, 4, 4, True), (129, 640, 300, 8, 4, True), (70, 160, 40, 8, 8, True), (33, 4096, 1000, 6, 6, False),
]


@pytest.mark.parametrize("n,d_in,d_out,bx,bw,asym", DP_GEMM)
def test_dp_linear_exact(n, d_in, d_out, bx, bw, asym):
    rng = np.random.default_rng(n * 7 + d_in + d_out + bx)
    qx = _rand_codes(rng, (n, d_in), bx, asym)
    qw = _rand_codes(rng, (d_out, d_in), bw, False)
    zx = rng.integers(0, 2 ** bx, n) if asym else None
    sx = rng.uniform(0.01, 2.0, n).astype(np.float32)
    sw = rng.uniform(0.001, 0.1, d_out).astype(np.float32)
    xp = torch.from_numpy(dp_planes.encode(qx, bx, asym)).to(DEV)
    wp = torch.from_numpy(dp_planes.encode(qw, bw, False)).to(DEV)
    np.testing.assert_array_equal(dp_planes.decode(xp.cpu().numpy()), qx)     # the test's own encoder
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    kw = {}
    if asym:
        kw = dict(x_zero=torch.from_numpy(zx.astype(np.int32)).to(DEV),
                  w_rowsum=torch.from_numpy(qw.sum(axis=1).astype(np.int32)).to(DEV))
    y = cat.cat_linear_dp(xp, bx, torch.from_numpy(sx).to(DEV), wp, bw, torch.from_numpy(sw).to(DEV), acc_out=acc, **kw)
    _, y_ref = O.w4a4_linear(qx, sx.astype(np.float64), qw, sw.astype(np.float64), zx=zx)
    acc_ref = O.int_gemm(qx - (zx[:, None] if asym else 0), qw)
    np.testing.assert_array_equal(acc.cpu().numpy(), acc_ref)
    assert rel_fro(y.cpu().numpy(), y_ref) < 1e-6
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("bx,bw,asym", [(8, 8, False), (8, 8, True), (6, 6, False)])
def test_dp_linear_extreme_accumulators(bx, bw, asym):
    """The largest codes over d_in = 65536 (the bound): every accumulator at its int32 limit range."""
    n, d_in, d_out = 8, 65536, 64
    qmx = 2 ** (bx - 1) - 1
    qx = np.full((n, d_in), 2 ** bx - 1 if asym else qmx, dtype=np.int64)
    if not asym:
        qx[1::2] = -qmx
    qmw = 2 ** (bw - 1) - 1
    qw = np.full((d_out, d_in), qmw, dtype=np.int64)
    qw[3, : d_in // 2] = -qmw
    qw[5, -300:] = np.arange(300) % 3 - 1
    zx = np.zeros(n, dtype=np.int64) if asym else None
    if asym:
        zx[1] = 2 ** bx - 1                          # (q - z) = 0 for every element of token 1
    ones = torch.ones(max(n, d_out), dtype=torch.float32, device=DEV)
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    kw = {}
    if asym:
        kw = dict(x_zero=torch.from_numpy(zx.astype(np.int32)).to(DEV),
                  w_rowsum=torch.from_numpy(qw.sum(axis=1).astype(np.int32)).to(DEV))
    cat.cat_linear_dp(torch.from_numpy(dp_planes.encode(qx, bx, asym)).to(DEV), bx, ones[:n].contiguous(),
                      torch.from_numpy(dp_planes.encode(qw, bw, False)).to(DEV), bw, ones[:d_out].contiguous(),
                      acc_out=acc, **kw)
    ref = O.int_gemm(qx - (zx[:, None] if asym else 0), qw)
    np.testing.assert_array_equal(acc.cpu().numpy(), ref)


# ------------------------------------------------------------------------------------------
# cat_transform_quantize_act_dp / cat_quantize_weights_dp against the oracle
# ------------------------------------------------------------------------------------------

def _cat_T(rng, d, k):
    X = rng.standard_normal((4 * k + 64, d)) @ (rng.standard_normal((d, d)) / np.sqrt(d) + np.eye(d))
    W = rng.standard_normal((d + 32, d)) * 0.02
    T, _ = O.build_transform("cat", d, k, O.calib_cov_block_sums(X, k) / X.shape[0], O.weight_autocorr_blocks(W, k))
    return T.astype(np.float32)


@pytest.mark.parametrize("n,d,k,dtype,bits,asym", [(130, 256, 32, "f32", 8, False), (200, 512, 128, "bf16", 6, False),
                                                   (67, 384, 64, "bf16", 3, False), (300, 256, 32, "bf16", 4, True),
                                                   (150, 512, 256, "f32", 8, True), (64, 64, 16, "bf16", 2, True)])
def test_dp_transform_quantize_act(n, d, k, dtype, bits, asym):
    rng = np.random.default_rng(n + d + bits)
    X = rng.standard_normal((n, d)) * rng.lognormal(0, 1.0, d) + (0.3 if asym else 0.0)
    X[0] = 0.0
    X[1] = 0.0
    X[1, d // 3] = 3.0
    X[2] *= 1e4
    Xt = WL.cast(X, dtype)
    T32 = _cat_T(rng, d, k)
    planes, sx, zx = cat.cat_transform_quantize_act_dp(to_dev(Xt), torch.from_numpy(T32).to(DEV), k, bits, asym)
    ref = O.transform_quantize_act(Xt.values, T32.astype(np.float64), bits=bits, asymmetric=asym)
    q = dp_planes.decode(planes.cpu().numpy())
    check_codes(q, ref.qx, ref.pre_x)
    np.testing.assert_allclose(sx.cpu().numpy().astype(np.float64), ref.sx, rtol=1e-5, atol=0)
    if asym:
        zg = zx.cpu().numpy()
        assert np.sum(zg != ref.zx) <= max(1, 1e-3 * n)
    assert sx[0].item() == 0.0 and np.all(q[0] == 0)
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("bits,asym", [(8, False), (6, False), (4, True), (8, True), (2, True)])
def test_dp_code_decision_exact_under_identity(bits, asym):
    """T = I: the codes are the definition's, exactly (bf16 inputs, ties included)."""
    rng = np.random.default_rng(3 * bits + asym)
    n, d, k = 300, 512, 64
    X = rng.integers(-120, 121, (n, d)) / 64.0 + (0.5 if asym else 0.0)      # many exact ties
    X[5] *= 2.0 ** -90
    Xt = WL.cast(X, "bf16")
    assert np.array_equal(Xt.values, X)
    T = np.tile(np.eye(k, dtype=np.float32), (d // k, 1, 1))
    planes, sx, zx = cat.cat_transform_quantize_act_dp(to_dev(Xt), torch.from_numpy(T).to(DEV), k, bits, asym)
    if asym:
        q, s, z, _ = O.quantize_rows_asymmetric(Xt.values, bits)
        np.testing.assert_array_equal(zx.cpu().numpy(), z)
    else:
        q, s, _ = O.quantize_rows_symmetric(Xt.values, bits)
    np.testing.assert_array_equal(dp_planes.decode(planes.cpu().numpy()), q)
    np.testing.assert_allclose(sx.cpu().numpy().astype(np.float64), s, rtol=1e-6, atol=0)


@pytest.mark.parametrize("kind,bits,l24", [("identity", 8, False), ("cat", 6, False), ("cat", 4, True),
                                            ("rht", 8, True), ("identity", 3, True)])
def test_dp_quantize_weights(kind, bits, l24):
    cfg = WL.small_config("dpw", d_in=512, d_out=300, n_eval=64, n_calib=512, k=64, seed=41)
    L = WL.make_layer(cfg)
    W, xc = to_dev(L.W), to_dev(L.x_calib)
    sig = cat.cat_calib_cov(xc, cfg.k) if kind == "cat" else None
    T, planes, sw, rs = cat.cat_quantize_weights_dp(W, cfg.k, kind, bits, sigma_x=sig, n_calib=cfg.n_calib,
                                                    rht_signs=L.rht_signs if kind == "rht" else None, l24_range=l24,
                                                    rowsum=True)
    ref = O.prepare_weights(L.W.values, kind, cfg.k, X_calib=L.x_calib.values, signs=L.rht_signs, bits=bits,
                            w_range="l2.4" if l24 else "max")
    q = dp_planes.decode(planes.cpu().numpy())
    np.testing.assert_array_equal(rs.cpu().numpy(), q.sum(axis=1))
    swg = sw.cpu().numpy().astype(np.float64)
    same = np.ones(q.shape[0], dtype=bool)
    if l24:
        # the chosen candidate per row: from the step, s = max|w'| (100 - i) / 100 / qmax
        qmax = 2 ** (bits - 1) - 1
        amax = np.max(np.abs(ref.Wt), axis=1)
        i_gpu = np.rint((1.0 - swg * qmax / amax) * 100).astype(int)
        i_ref = ref.shrink
        same = i_gpu == i_ref
        if not same.all():
            scores = O.weight_range_lp(ref.Wt, bits, return_scores=True)[1]
            rows = np.where(~same)[0]
            a, b = scores[rows, i_gpu[rows]], scores[rows, i_ref[rows]]
            assert np.all(np.abs(a - b) <= 1e-5 * np.maximum(a, b)), "a different range away from a near-tie"
        assert same.mean() > 0.95
    check_codes(q[same], ref.qw[same], ref.pre_w[same])
    np.testing.assert_allclose(swg[same], ref.sw[same], rtol=1e-5)
    if kind == "identity" and not l24:
        np.testing.assert_array_equal(q, ref.qw)
    assert cat.cat_device_status()[0] == 0


# ------------------------------------------------------------------------------------------
# Whole layer at other bit widths and with Sec. 6's quantizer
# ------------------------------------------------------------------------------------------

def gpu_layer_dp(L, kind, k, bx, bw, asym, l24):
    x, W, xc = to_dev(L.x_eval), to_dev(L.W), to_dev(L.x_calib)
    sig = cat.cat_calib_cov(xc, k) if kind == "cat" else None
    T, wp, sw, rs = cat.cat_quantize_weights_dp(W, k, kind, bw, sigma_x=sig, n_calib=L.cfg.n_calib,
                                                rht_signs=L.rht_signs if kind == "rht" else None, l24_range=l24,
                                                rowsum=asym)
    xp, sx, zx = cat.cat_transform_quantize_act_dp(x, T, k, bx, asym)
    return cat.cat_linear_dp(xp, bx, sx, wp, bw, sw, x_zero=zx, w_rowsum=rs), sw


def reconcile_ranges(ref, sw_gpu, bits):
    """The L_2.4 search may choose another candidate than the oracle where the two candidates' scores
    agree to 1e-5 (either is a correct result): check that, then redo the oracle's weight codes and
    output with the library's choice in those rows."""
    pw = ref["prep"]
    qmax = 2 ** (bits - 1) - 1
    amax = np.max(np.abs(pw.Wt), axis=1)
    nz = amax > 0
    i_gpu = np.zeros(len(amax), dtype=int)
    i_gpu[nz] = np.rint((1.0 - sw_gpu[nz] * qmax / amax[nz]) * 100).astype(int)
    i_ref = pw.shrink
    rows = np.where(i_gpu != i_ref)[0]
    if len(rows) == 0:
        return ref["y_hat"], 0
    scores = O.weight_range_lp(pw.Wt, bits, return_scores=True)[1]
    a, b = scores[rows, i_gpu[rows]], scores[rows, i_ref[rows]]
    assert np.all(np.abs(a - b) <= 1e-5 * np.maximum(a, b)), "a different range away from a near-tie"
    qw, swr, _ = O.quantize_rows_symmetric(pw.Wt, bits, shrink=i_gpu)
    ac = ref["act"]
    _, y_hat = O.w4a4_linear(ac.qx, ac.sx, qw, swr, zx=ac.zx)
    return y_hat, len(rows)


LAYERS = [
    WL.small_config("dp_bf16_k128", d_in=512, d_out=384, n_eval=300, n_calib=512, k=128, seed=51),
    WL.small_config("dp_swiglu_k64", d_in=768, d_out=200, n_eval=70, n_calib=256, k=64, act="swiglu", seed=52),
]


@pytest.mark.parametrize("cfg", LAYERS, ids=lambda c: c.name)
@pytest.mark.parametrize("kind", ["identity", "cat"])
@pytest.mark.parametrize("bx,bw,asym,l24", [(4, 4, False, False), (8, 4, False, False), (6, 6, False, False),
                                            (8, 8, False, False), (4, 4, True, True), (8, 8, True, True)])
def test_dp_layer_end_to_end(cfg, kind, bx, bw, asym, l24):
    L = WL.make_layer(cfg)
    y, sw = gpu_layer_dp(L, kind, cfg.k, bx, bw, asym, l24)
    y = y.cpu().numpy()
    ref = O.cat_layer(L.x_eval.values, L.W.values, kind, cfg.k, X_calib=L.x_calib.values, bits_x=bx, bits_w=bw,
                      act_asym=asym, w_range="l2.4" if l24 else "max")
    y_hat = ref["y_hat"]
    if l24:
        y_hat, _ = reconcile_ranges(ref, sw.cpu().numpy().astype(np.float64), bw)
    assert rel_fro(y, y_hat) < 1e-3
    sig, err = O.sqnr_sums(ref["y"], y_hat)
    s3 = cat.cat_sqnr(torch.from_numpy(ref["y"].astype(np.float32)).to(DEV), torch.from_numpy(y).to(DEV)).cpu().numpy()
    assert abs(s3[2] - 10 * np.log10(sig / err)) < 0.01, (s3[2], 10 * np.log10(sig / err))
    assert cat.cat_device_status()[0] == 0


def test_dp_w4a4_equals_packed_path():
    """The packed W4A4 path's own codes and steps, re-encoded as one digit plane each, give the same y
    through the digit-plane GEMM bit for bit (both GEMMs accumulate exactly and scale alike)."""
    import sm4x8
    cfg = LAYERS[0]
    L = WL.make_layer(cfg)
    x, W, xc = to_dev(L.x_eval), to_dev(L.W), to_dev(L.x_calib)
    sig = cat.cat_calib_cov(xc, cfg.k)
    T, Wq, sw = cat.cat_quantize_weights(W, cfg.k, "cat", sigma_x=sig, n_calib=cfg.n_calib)
    xq, sx = cat.cat_transform_quantize_act(x, T, cfg.k)
    y_packed = cat.cat_w4a4_linear(xq, sx, Wq, sw)
    qx, qw = sm4x8.unpack(xq.cpu().numpy()), sm4x8.unpack(Wq.cpu().numpy())
    xp = torch.from_numpy(dp_planes.encode(qx, 4, False)).to(DEV)
    wp = torch.from_numpy(dp_planes.encode(qw, 4, False)).to(DEV)
    y_dp = cat.cat_linear_dp(xp, 4, sx, wp, 4, sw)
    assert torch.equal(y_dp, y_packed)
