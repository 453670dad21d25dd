"""Parity of the CUDA path (through the C ABI) with the fp64 CPU oracle, element by element.

Tolerances (the benchmark spec's targets, applied per call):
* integer accumulators: bit-exact given identical codes;
* INT4 codes: may differ by +-1, in at most 1e-4 of the elements (at least one element is
  allowed in small cases), and only where the oracle's pre-rounding value lies within 1e-5
  (relative) of a rounding boundary -- the GPU accumulates x' = T x in fp32;
* steps s_x, s_w: 1e-5 relative; y: 1e-3 relative Frobenius; SQNR: 0.01 dB;
* calibration sums: fp32 rows 1e-10 relative Frobenius (compensated accumulation); bf16 rows 1e-6
  (tensor-core fp32 accumulation: ~1e-7 measured, bounded by ~n 2^-24 per entry);
* transform blocks: fp32 layers 1e-6 relative (fp32 storage of the float64 construction); bf16
  layers 1e-5 (fp32 calibration sums, ~1e-7, times the sensitivity of T to Sigma_x: ~4 on the
  layer configurations, ~20 on the strongly low-rank small test layer).  The binding checks
  stay the codes (+-1 within 1e-5 of a boundary), y and SQNR.
"""
import numpy as np
import pytest
import torch

import oracle as O
import sm4x8
import workloads as WL

pytestmark = pytest.mark.gpu

cat = pytest.importorskip("paper_2603_04359_gb300")
DEV = "cuda"


def to_dev(t: WL.Tensor) -> torch.Tensor:
    if t.dtype == "f32":
        return torch.from_numpy(np.ascontiguousarray(t.raw)).to(DEV)
    return torch.from_numpy(np.ascontiguousarray(t.raw).view(np.int16)).view(torch.bfloat16).to(DEV)


def check_codes(q_gpu, q_ref, pre_ref, rel=1e-5, frac=1e-4):
    q_gpu = np.asarray(q_gpu)
    diff = q_gpu - q_ref
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


# ------------------------------------------------------------------------------------------
# cat_calib_cov
# ------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,d,k,dtype", [(77, 256, 32, "f32"), (300, 512, 128, "bf16"), (1000, 512, 256, "bf16"),
                                         (64, 64, 16, "f32"), (513, 384, 64, "bf16"), (70, 96, 32, "bf16"),
                                         (200, 160, 16, "bf16"), (5000, 256, 128, "bf16")])
def test_calib_cov(n, d, k, dtype):
    rng = np.random.default_rng(n + d)
    X = rng.standard_normal((n, d)) * rng.lognormal(0, 1.5, d)
    Xt = WL.cast(X, dtype)
    tol = 1e-10 if dtype == "f32" else 1e-6
    S = cat.cat_calib_cov(to_dev(Xt), k).cpu().numpy()
    ref = O.calib_cov_block_sums(Xt.values, k)
    assert rel_fro(S, ref) < tol
    # accumulate a second batch
    X2 = WL.cast(rng.standard_normal((n // 2 + 1, d)), dtype)
    out = torch.from_numpy(S).to(DEV)
    cat.cat_calib_cov(to_dev(X2), k, out=out, accumulate=True)
    ref2 = O.calib_cov_block_sums(np.vstack([Xt.values, X2.values]), k)
    assert rel_fro(out.cpu().numpy(), ref2) < tol


# ------------------------------------------------------------------------------------------
# cat_transform_quantize_act (given the same transform)
# ------------------------------------------------------------------------------------------

def _cat_T(rng, d, k):
    X = rng.standard_normal((4 * k + 64, d)) @ (rng.standard_normal((d, d)) / np.sqrt(d) + np.eye(d))
    W = rng.standard_normal((d + 32, d)) * 0.02
    T, _ = O.build_transform("cat", d, k, O.calib_cov_block_sums(X, k) / X.shape[0], O.weight_autocorr_blocks(W, k))
    return T.astype(np.float32)


@pytest.mark.parametrize("n,d,k,dtype", [(130, 256, 32, "f32"), (67, 384, 128, "bf16"), (200, 512, 256, "bf16"),
                                         (5, 64, 16, "bf16"), (300, 1024, 64, "f32"), (300, 1024, 64, "bf16"),
                                         (300, 640, 128, "bf16"), (1000, 256, 128, "bf16"),
                                         # more units per CTA than tensor memory holds: the fused kernel
                                         # in waves (5 and 11 units per CTA, ragged last tile)
                                         (2560, 4096, 128, "bf16"), (1300, 8192, 64, "bf16"),
                                         # k < 128 block-diagonal inside 128-channel groups (one wave, waves)
                                         (300, 512, 32, "bf16"), (130, 384, 16, "bf16"), (2560, 4096, 32, "bf16"),
                                         (1100, 10240, 64, "bf16"),
                                         # 64 | d but not 128: the 64-wide kernels (one wave, two passes)
                                         (300, 192, 64, "bf16"), (1100, 9920, 64, "bf16"),
                                         # more groups than SMs and more than one wave: two passes
                                         (520, 20480, 128, "bf16"),
                                         # k = 256: 64-output quarters of a block over its 256 inputs
                                         # (one wave, waves, contiguous ranges; beyond: the SIMT kernel)
                                         (2560, 2048, 256, "bf16"), (2560, 4096, 256, "bf16"),
                                         (300, 10240, 256, "bf16"), (1300, 10240, 256, "bf16")])
def test_transform_quantize_act(n, d, k, dtype):
    rng = np.random.default_rng(7 * n + d)
    X = rng.standard_normal((n, d)) * rng.lognormal(0, 1.0, d)
    X[0] = 0.0                       # all-zero token
    X[1] = 0.0
    X[1, d // 3] = 3.0               # one-hot token
    X[2] *= 1e4                      # a huge token
    Xt = WL.cast(X, dtype)
    T32 = _cat_T(rng, d, k)
    xq, sx = cat.cat_transform_quantize_act(to_dev(Xt), torch.from_numpy(T32).to(DEV), k)
    ref = O.transform_quantize_act(Xt.values, T32.astype(np.float64))
    q = sm4x8.unpack(xq.cpu().numpy())
    check_codes(q, ref.qx, ref.pre_x)
    sxg = sx.cpu().numpy().astype(np.float64)
    assert sxg[0] == 0.0 and np.all(q[0] == 0)
    np.testing.assert_allclose(sxg, ref.sx, rtol=1e-5, atol=0)
    assert np.abs(q).max() == 7
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("n,d,k,dtype", [(67, 384, 128, "bf16"), (300, 1024, 64, "bf16"), (1000, 256, 128, "bf16"),
                                         (2560, 4096, 128, "bf16"), (1300, 8192, 64, "bf16"),
                                         (300, 512, 32, "bf16"), (130, 384, 16, "bf16"), (300, 192, 64, "bf16"),
                                         (1100, 9920, 64, "bf16"), (200, 512, 256, "bf16"), (2560, 4096, 256, "bf16"),
                                         (130, 256, 32, "f32")])
def test_transform_with_presplit_planes_is_identical(n, d, k, dtype):
    """T's bf16 planes split once (cat_split_transform) and bulk-copied by the kernels give the same
    codes and steps, bit for bit, as the kernels' own split (fused, two-pass, and the SIMT path that
    ignores the planes)."""
    rng = np.random.default_rng(5 * n + d)
    X = WL.cast(rng.standard_normal((n, d)) * rng.lognormal(0, 1.0, d), dtype)
    T32 = torch.from_numpy(_cat_T(rng, d, k)).to(DEV)
    planes = cat.cat_split_transform(T32, k) if (dtype == "bf16" and cat.cat_split_transform_bytes(d, k) > 0) else None
    xq0, sx0 = cat.cat_transform_quantize_act(to_dev(X), T32, k)
    xq1, sx1 = cat.cat_transform_quantize_act_split(to_dev(X), T32, planes, k)
    assert torch.equal(xq0, xq1) and torch.equal(sx0, sx1)
    assert cat.cat_device_status()[0] == 0


def test_nonfinite_activation_reports_numeric():
    d, k = 128, 32
    X = np.ones((70, d), dtype=np.float32)
    X[3, 5] = np.inf
    T = np.tile(np.eye(k, dtype=np.float32), (d // k, 1, 1))
    cat.cat_device_status()  # clear
    xq, sx = cat.cat_transform_quantize_act(torch.from_numpy(X).to(DEV), torch.from_numpy(T).to(DEV), k)
    st, word = cat.cat_device_status()
    assert st == 4 and word & 2
    assert sx[3].item() == 0.0
    assert sx[4].item() == pytest.approx(1.0 / 7.0, rel=1e-6)
    assert cat.cat_device_status()[0] == 0  # cleared


@pytest.mark.parametrize("n,d,k", [(2560, 4096, 128),    # the fused kernel in waves
                                   (1100, 9920, 64),     # the two-pass kernel (64-wide)
                                   (2560, 4096, 32),     # waves, k = 32 block-diagonal in 128-channel groups
                                   (2560, 4096, 256)])   # waves, k = 256 in 64-output quarters
def test_nonfinite_activation_many_units(n, d, k):
    """bf16 rows with more units per CTA than tensor memory holds: a row holding inf or NaN gets step 0
    and all codes 0, the status reports it, and the other rows are unaffected."""
    rng = np.random.default_rng(11)
    X = rng.standard_normal((n, d))
    Xt = WL.cast(X, "bf16")
    raw = Xt.raw.copy()
    raw[5, 17] = 0x7F80                     # +inf
    raw[900, d - 96] = 0x7FC0               # NaN
    bad = WL.Tensor(values=WL.bf16_bits_to_f32(raw), raw=raw, dtype="bf16")
    T32 = _cat_T(rng, d, k)
    cat.cat_device_status()  # clear
    xq, sx = cat.cat_transform_quantize_act(to_dev(bad), torch.from_numpy(T32).to(DEV), k)
    st, word = cat.cat_device_status()
    assert st == 4 and word & 2
    q = sm4x8.unpack(xq.cpu().numpy())
    sxg = sx.cpu().numpy()
    for r in (5, 900):
        assert sxg[r] == 0.0 and np.all(q[r] == 0)
    good = np.ones(n, dtype=bool)
    good[[5, 900]] = False
    ref = O.transform_quantize_act(Xt.values[good], T32.astype(np.float64))
    check_codes(q[good], ref.qx, ref.pre_x)
    np.testing.assert_allclose(sxg[good].astype(np.float64), ref.sx, rtol=1e-5, atol=0)
    assert cat.cat_device_status()[0] == 0


def _bf16_tie_pairs():
    """For every bf16 step a in [1, 2): the bf16 values v in [a/14, a] with 7 v / a exactly a
    half-integer (exact rational arithmetic)."""
    from fractions import Fraction
    out = {}
    for ma in range(128):
        a = Fraction(128 + ma, 128)
        vs = []
        for e in range(-4, 1):
            for mv in range(128):
                v = Fraction(128 + mv, 128) * Fraction(2) ** e
                t = 7 * v / a
                if v <= a and t.denominator == 2:
                    vs.append(float(v))
        if vs:
            out[float(a)] = vs
    return out


def _tie_rows(rng, n, d):
    """bf16-representable rows in which many entries make 7 v / max|v| an exact half-integer, at
    ordinary scales and at scales that take the rescaled route (2^-100, 2^110)."""
    pairs = _bf16_tie_pairs()
    steps = np.array(sorted(pairs))
    X = np.empty((n, d))
    for r in range(n):
        a = float(rng.choice(steps))
        ties = np.array(pairs[a])
        row = WL.cast(rng.uniform(-a, a, d) * 0.99, "bf16").values.astype(np.float64)  # ordinary values
        pick = rng.random(d) < 0.5
        row[pick] = rng.choice(ties, pick.sum()) * rng.choice([-1.0, 1.0], pick.sum())
        row[rng.integers(d)] = a * rng.choice([-1.0, 1.0])
        scale = {0: 2.0 ** -100, 1: 2.0 ** 110}.get(r, 2.0 ** int(rng.integers(-12, 12)))
        X[r] = row * scale
    Xt = WL.cast(X, "bf16")
    assert np.array_equal(Xt.values, X)                        # every value is a bf16 number
    return X


@pytest.mark.parametrize("n,d,k,dtype", [(300, 512, 64, "bf16"), (1000, 1024, 128, "bf16"),   # fused
                                         (2560, 4096, 128, "bf16"),                            # waves
                                         (1100, 9920, 64, "bf16"),                             # two-pass
                                         (300, 512, 32, "bf16"),                               # k = 32 in groups
                                         (200, 512, 256, "bf16"),                              # k = 256
                                         (130, 256, 32, "f32"),                                # SIMT
                                         (70, 64, 16, "bf16")])
def test_code_decision_exact_on_ties(n, d, k, dtype):
    """With T = I the transformed row is the input row, so the codes must equal the definition's
    round-half-to-even of 7 v / max|v| exactly, ties included (Lemma 2 range, Sec. 6 RTN).  The rows
    are built so that a float32 reciprocal-multiply decision would get many of them wrong."""
    rng = np.random.default_rng(n + k)
    X = _tie_rows(rng, n, d)
    Xt = WL.cast(X, dtype)
    ref = O.quantize_rows_symmetric(Xt.values)
    a32 = np.max(np.abs(Xt.values), axis=1).astype(np.float32)
    q32 = np.clip(np.rint(Xt.values.astype(np.float32) * (np.float32(7) / a32)[:, None]), -7, 7)
    assert np.sum(q32 != ref[0]) > 10                          # the fixture has teeth
    T = np.tile(np.eye(k, dtype=np.float32), (d // k, 1, 1))
    xq, sx = cat.cat_transform_quantize_act(to_dev(Xt), torch.from_numpy(T).to(DEV), k)
    np.testing.assert_array_equal(sm4x8.unpack(xq.cpu().numpy()), ref[0])
    np.testing.assert_allclose(sx.cpu().numpy().astype(np.float64), ref[1], rtol=1e-6, atol=0)
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("k", [32, 128])
def test_weight_code_decision_exact_on_ties(k):
    """Weight preparation with T = I quantizes the rows of W itself: exact codes, ties included."""
    rng = np.random.default_rng(99 + k)
    W = _tie_rows(rng, 300, 1024)
    Wt = WL.cast(W, "bf16")
    T, Wq, sw = cat.cat_quantize_weights(to_dev(Wt), k, "identity")
    ref = O.quantize_rows_symmetric(Wt.values)
    np.testing.assert_array_equal(sm4x8.unpack(Wq.cpu().numpy()), ref[0])
    np.testing.assert_allclose(sw.cpu().numpy().astype(np.float64), ref[1], rtol=1e-6, atol=0)
    assert cat.cat_device_status()[0] == 0


# ------------------------------------------------------------------------------------------
# cat_w4a4_linear (given identical codes): exact accumulators
# ------------------------------------------------------------------------------------------

GEMM_SHAPES = [
    # n <= 32: tcgen05 weight streaming, tokens resident in shared memory (the last five walk many
    # 128-row units per CTA, the last two with few packed stages beside a large token operand)
    (1, 64, 8), (5, 160, 100), (17, 96, 33), (16, 4096, 520), (32, 384, 300), (8, 8192, 200),
    (24, 2048, 1000), (2, 1024, 17), (3, 4096, 20000), (20, 2048, 40000), (9, 8192, 12000),
    (16, 9216, 300), (32, 4608, 260),
    # more 128-row units than SMs: the (unit, K step) sequence cut into equal ranges (stream-K), units
    # cut between CTAs combined exactly; K steps per row not a multiple of the four decode groups
    (16, 1536, 20000), (32, 4608, 19500),
    (3, 12288, 100),                                  # n <= 32, tokens too large for shared memory: mma.sync
    (33, 128, 256), (128, 256, 256), (129, 160, 300), (300, 384, 520), (257, 4096, 64),  # tcgen05 path
    (512, 1024, 1024), (1024, 512, 6144),                                                # ... several tiles per pair
    (256, 1024, 9984), (300, 2048, 5030),  # a last wave of 2 / 4 tiles on 76 pairs, split along K into 4 / 8 parts
]


@pytest.mark.parametrize("n,d_in,d_out", GEMM_SHAPES)
def test_w4a4_linear_exact(n, d_in, d_out):
    rng = np.random.default_rng(n * 1000 + d_in + d_out)
    qx = WL.random_codes(rng, (n, d_in)).astype(np.int64)
    qw = WL.random_codes(rng, (d_out, d_in)).astype(np.int64)
    sx = rng.uniform(0.01, 2.0, n).astype(np.float32)
    sw = rng.uniform(0.001, 0.1, d_out).astype(np.float32)
    xq = torch.from_numpy(sm4x8.pack(qx)).to(DEV)
    wq = torch.from_numpy(sm4x8.pack(qw)).to(DEV)
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    y = cat.cat_w4a4_linear(xq, torch.from_numpy(sx).to(DEV), wq, torch.from_numpy(sw).to(DEV), acc_out=acc)
    ref_acc = O.int_gemm(qx, qw)
    np.testing.assert_array_equal(acc.cpu().numpy(), ref_acc)
    ref_y = O.dequantize_output(ref_acc, sx.astype(np.float64), sw.astype(np.float64))
    assert rel_fro(y.cpu().numpy(), ref_y) < 1e-6
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("n,d_in", [(8, 14336), (200, 14336), (16, 4096)])
def test_w4a4_linear_extreme_accumulators(n, d_in):
    d_out = 64
    qx = np.full((n, d_in), 7, dtype=np.int64)
    qx[1::2] = -7
    qw = np.full((d_out, d_in), 7, dtype=np.int64)
    qw[3, : d_in // 2] = -7                       # cancels to zero
    qw[5, -300:] = np.arange(300) % 3 - 1         # small codes after a large prefix
    ones = torch.ones(max(n, d_out), dtype=torch.float32, device=DEV)
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    cat.cat_w4a4_linear(torch.from_numpy(sm4x8.pack(qx)).to(DEV), ones[:n].contiguous(),
                        torch.from_numpy(sm4x8.pack(qw)).to(DEV), ones[:d_out].contiguous(), acc_out=acc)
    ref = O.int_gemm(qx, qw)
    assert np.abs(ref).max() == 49 * d_in
    np.testing.assert_array_equal(acc.cpu().numpy(), ref)


# ------------------------------------------------------------------------------------------
# cat_w4a4_linear_sqnr: the GEMM with the SQNR sums formed in its epilogue
# ------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,d_in,d_out", [(300, 1024, 520), (513, 512, 256), (257, 4096, 130), (16, 1024, 200),
                                          (129, 160, 300), (24, 2048, 40000), (16, 9216, 300), (3, 12288, 100),
                                          (1024, 512, 6144),    # several pair tiles per CTA pair
                                          (300, 2048, 5032)])   # a split last wave
def test_w4a4_linear_sqnr_fused(n, d_in, d_out):
    """y equals cat_w4a4_linear's bit for bit; the sums match the oracle's over the same outputs
    (fused in the GEMM epilogue for n > 32 with d_out % 4 == 0 and in the tcgen05 decode kernel,
    else the separate reduction)."""
    rng = np.random.default_rng(n + 7 * d_in + 13 * d_out)
    qx = WL.random_codes(rng, (n, d_in)).astype(np.int64)
    qw = WL.random_codes(rng, (d_out, d_in)).astype(np.int64)
    sx = rng.uniform(0.01, 2.0, n).astype(np.float32)
    sw = rng.uniform(0.001, 0.1, d_out).astype(np.float32)
    xq = torch.from_numpy(sm4x8.pack(qx)).to(DEV)
    wq = torch.from_numpy(sm4x8.pack(qw)).to(DEV)
    sx_d, sw_d = torch.from_numpy(sx).to(DEV), torch.from_numpy(sw).to(DEV)
    y_plain = cat.cat_w4a4_linear(xq, sx_d, wq, sw_d)
    y_ref = (y_plain.double() + torch.randn(n, d_out, device=DEV, dtype=torch.float64) * 0.05).float().contiguous()
    for rep in range(2):                                   # twice: the sums restart from zero each call
        y, out3 = cat.cat_w4a4_linear_sqnr(xq, sx_d, wq, sw_d, y_ref)
        assert torch.equal(y, y_plain)
        sig, err = O.sqnr_sums(y_ref.cpu().numpy(), y.cpu().numpy())
        o = out3.cpu().numpy()
        assert abs(o[0] - sig) <= 1e-6 * sig and abs(o[1] - err) <= 1e-6 * err
        assert abs(o[2] - 10 * np.log10(sig / err)) < 1e-5
    assert cat.cat_device_status()[0] == 0


# ------------------------------------------------------------------------------------------
# cat_sqnr
# ------------------------------------------------------------------------------------------

@pytest.mark.parametrize("numel", [1, 7, 4096, 1_000_003])
def test_sqnr(numel):
    rng = np.random.default_rng(numel)
    y = rng.standard_normal(numel).astype(np.float32) * 3
    yh = (y + rng.standard_normal(numel).astype(np.float32) * 0.05).astype(np.float32)
    out = cat.cat_sqnr(torch.from_numpy(y).to(DEV), torch.from_numpy(yh).to(DEV)).cpu().numpy()
    sig, err = O.sqnr_sums(y, yh)
    assert abs(out[0] - sig) <= 1e-6 * sig and abs(out[1] - err) <= 1e-6 * err
    assert abs(out[2] - 10 * np.log10(sig / err)) < 1e-5


# ------------------------------------------------------------------------------------------
# Whole layer: library pipeline vs oracle pipeline from the same raw inputs
# ------------------------------------------------------------------------------------------

def gpu_layer(L: WL.Layer, kind: str, k: int):
    x, W, xc = to_dev(L.x_eval), to_dev(L.W), to_dev(L.x_calib)
    sig = cat.cat_calib_cov(xc, k) if kind == "cat" else None
    T, Wq, sw = cat.cat_quantize_weights(W, k, kind, sigma_x=sig, n_calib=L.cfg.n_calib,
                                         rht_signs=L.rht_signs if kind == "rht" else None)
    xq, sx = cat.cat_transform_quantize_act(x, T, k)
    y = cat.cat_w4a4_linear(xq, sx, Wq, sw)
    return dict(sigma=sig, T=T, Wq=Wq, sw=sw, xq=xq, sx=sx, y=y)


SMALL = [
    WL.CONFIGS["c1_256x256_k32_f32"],
    WL.small_config("s_bf16_k128", d_in=512, d_out=384, n_eval=300, n_calib=512, k=128, seed=21),
    WL.small_config("s_swiglu_k64", d_in=768, d_out=200, n_eval=70, n_calib=256, k=64, act="swiglu", seed=22),
    WL.small_config("s_decode_k256", d_in=512, d_out=1000, n_eval=16, n_calib=600, k=256, seed=23),
]


@pytest.mark.parametrize("cfg", SMALL, ids=lambda c: c.name)
@pytest.mark.parametrize("kind", ["identity", "rht", "cat"])
def test_layer_end_to_end(cfg, kind):
    L = WL.make_layer(cfg)
    k = cfg.k
    g = gpu_layer(L, kind, k)
    ref = O.cat_layer(L.x_eval.values, L.W.values, kind, k, X_calib=L.x_calib.values, signs=L.rht_signs)
    # transform blocks
    assert rel_fro(g["T"].cpu().numpy(), ref["prep"].T) < (1e-6 if cfg.dtype == "f32" else 1e-5)
    # weight and activation codes, steps (T = I: the quantizer sees the inputs themselves, exact codes)
    if kind == "identity":
        np.testing.assert_array_equal(sm4x8.unpack(g["Wq"].cpu().numpy()), ref["prep"].qw)
        np.testing.assert_array_equal(sm4x8.unpack(g["xq"].cpu().numpy()), ref["act"].qx)
    check_codes(sm4x8.unpack(g["Wq"].cpu().numpy()), ref["prep"].qw, ref["prep"].pre_w)
    np.testing.assert_allclose(g["sw"].cpu().numpy(), ref["prep"].sw, rtol=1e-5)
    check_codes(sm4x8.unpack(g["xq"].cpu().numpy()), ref["act"].qx, ref["act"].pre_x)
    np.testing.assert_allclose(g["sx"].cpu().numpy(), ref["act"].sx, rtol=1e-5)
    # output and SQNR (y_ref in fp32, as the benchmark supplies it)
    y_hat = g["y"].cpu().numpy()
    assert rel_fro(y_hat, ref["y_hat"]) < 1e-3
    y_ref = torch.from_numpy(ref["y"].astype(np.float32)).to(DEV)
    s3 = cat.cat_sqnr(y_ref, g["y"]).cpu().numpy()
    assert abs(s3[2] - ref["sqnr_db"]) < 0.01
    assert cat.cat_device_status()[0] == 0


# ------------------------------------------------------------------------------------------
# The gate/up layer's sweep, reduced: every block size x every transform through the library
# ------------------------------------------------------------------------------------------

SWEEP_LAYER = WL.small_config("s_gateup_sweep", d_in=1024, d_out=1792, n_eval=384, n_calib=512, k=128,
                              outlier_frac=0.005, outlier_scale=200.0, w_std=0.01, seed=25)


@pytest.mark.parametrize("k", [32, 64, 128, 256])
def test_block_size_transform_sweep(k):
    """SQNR of identity, randomized Hadamard and CAT transforms at block size k (Sec. 4) matches the
    oracle's within 0.01 dB, and CAT beats both (Sec. 3-4: it raises concentration and alignment;
    with outlier channels this strong the rotation alone barely moves the SQNR)."""
    L = WL.make_layer(SWEEP_LAYER)
    res = {}
    for kind in ("identity", "rht", "cat"):
        g = gpu_layer(L, kind, k)
        ref = O.cat_layer(L.x_eval.values, L.W.values, kind, k, X_calib=L.x_calib.values, signs=L.rht_signs)
        y_ref = torch.from_numpy(ref["y"].astype(np.float32)).to(DEV)
        s3 = cat.cat_sqnr(y_ref, g["y"]).cpu().numpy()
        assert abs(s3[2] - ref["sqnr_db"]) < 0.01, (kind, s3[2], ref["sqnr_db"])
        res[kind] = float(s3[2])
    assert res["cat"] > res["rht"] + 10.0 and res["cat"] > res["identity"] + 10.0, res
    assert cat.cat_device_status()[0] == 0


# ------------------------------------------------------------------------------------------
# Per-layer diagnostics: concentration, alignment and the Theorem-1 prediction from the library's
# row statistics of x' = T x and W' = W T^{-1}
# ------------------------------------------------------------------------------------------

@pytest.mark.parametrize("cfg", SMALL + [SWEEP_LAYER], ids=lambda c: c.name)
@pytest.mark.parametrize("kind", ["identity", "rht", "cat"])
def test_layer_diagnostics(cfg, kind):
    """C(x') and C(W') (Lemmas 2 and 3), A(x', W') and the Theorem-1 SQNR from cat_block_row_stats
    match the oracle's analysis functions on the oracle's x' and W' within 1e-4 (fp32 products)."""
    L = WL.make_layer(cfg)
    k = cfg.k
    g = gpu_layer(L, kind, k)
    ref = O.cat_layer(L.x_eval.values, L.W.values, kind, k, X_calib=L.x_calib.values, signs=L.rht_signs)
    Xp = O.apply_act_transform(L.x_eval.values, ref["prep"].T)
    Wp = ref["prep"].Wt
    # the weight rows need T^{-1}: the inverse of the library's own T blocks, on the host
    Tinv = np.linalg.inv(g["T"].double().cpu().numpy()).astype(np.float32)
    xs, xa, x3 = cat.cat_block_row_stats(to_dev(L.x_eval), k, g["T"])
    ws, wa, w3 = cat.cat_block_row_stats(to_dev(L.W), k, torch.from_numpy(Tinv).to(DEV), transpose=True)
    x3, w3 = x3.cpu().numpy(), w3.cpu().numpy()
    np.testing.assert_allclose(xs.cpu().numpy(), np.sum(Xp * Xp, axis=1), rtol=1e-4, atol=1e-12)
    np.testing.assert_allclose(xa.cpu().numpy(), np.max(np.abs(Xp), axis=1), rtol=1e-4, atol=1e-12)
    np.testing.assert_allclose(ws.cpu().numpy(), np.sum(Wp * Wp, axis=1), rtol=1e-4, atol=1e-12)
    np.testing.assert_allclose(wa.cpu().numpy(), np.max(np.abs(Wp), axis=1), rtol=1e-4, atol=1e-12)
    c_x, c_w = x3[0] / x3[1], w3[0] / w3[1]
    assert abs(c_x / O.concentration_act(Xp) - 1) < 1e-4
    assert abs(c_w / O.concentration_weight(Wp) - 1) < 1e-4
    assert abs(x3[2] - 10 * np.log10(c_x)) < 1e-4
    y = O.linear(L.x_eval.values, L.W.values)
    sum_y2 = float(cat.cat_sqnr(torch.from_numpy(y.astype(np.float32)).to(DEV), g["y"]).cpu().numpy()[0])
    a = sum_y2 / (w3[0] * x3[0])
    assert abs(a / O.alignment(Xp, Wp) - 1) < 1e-4
    n2 = O.n_intervals(4) ** 2
    pred = 12.0 * O.parallel(n2 * c_x, n2 * c_w) * a
    assert abs(O.db(pred) - O.db(O.theorem1_sqnr(Xp, Wp))) < 1e-3
    # the two measured sides of Theorem 1 (Lemma 2: only activations quantized; Lemma 3: only weights)
    y_ref = torch.from_numpy(y.astype(np.float32)).to(DEV)
    act_db, w_db = cat.one_sided_sqnr(to_dev(L.x_eval), to_dev(L.W), k, g["T"], torch.from_numpy(Tinv).to(DEV),
                                      g["xq"], g["sx"], g["Wq"], g["sw"], y_ref)
    assert abs(act_db - O.db(O.sqnr_act_only(Xp, Wp))) < 0.01, (act_db, O.db(O.sqnr_act_only(Xp, Wp)))
    assert abs(w_db - O.db(O.sqnr_weight_only(Xp, Wp))) < 0.01, (w_db, O.db(O.sqnr_weight_only(Xp, Wp)))
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("rows,d,k,transpose,dtype", [(70, 256, 32, False, "f32"), (300, 512, 128, True, "bf16"),
                                                      (5, 64, 16, False, "bf16"), (129, 768, 256, True, "f32")])
def test_block_transform_and_dequantize(rows, d, k, transpose, dtype):
    rng = np.random.default_rng(rows + d)
    V = WL.cast(rng.standard_normal((rows, d)) * rng.lognormal(0, 1, d), dtype)
    M = (rng.standard_normal((d // k, k, k)) / np.sqrt(k)).astype(np.float32)
    out = cat.cat_block_transform(to_dev(V), k, torch.from_numpy(M).to(DEV), transpose=transpose).cpu().numpy()
    Mb = np.transpose(M, (0, 2, 1)) if transpose else M          # v'_b = M_b v_b, or M_b^T v_b
    ref = O.apply_act_transform(V.values, Mb.astype(np.float64))
    assert rel_fro(out, ref) < 1e-6
    q = WL.random_codes(rng, (rows, d)).astype(np.int64)
    s_ = rng.uniform(0.01, 1, rows).astype(np.float32)
    deq = cat.cat_dequantize_codes(torch.from_numpy(sm4x8.pack(q)).to(DEV), torch.from_numpy(s_).to(DEV)).cpu().numpy()
    np.testing.assert_array_equal(deq, (q * s_[:, None].astype(np.float64)).astype(np.float32))


@pytest.mark.parametrize("m,n,kd", [(1, 1, 1), (130, 257, 96), (512, 384, 1024), (33, 1000, 17)])
def test_gemm_f32(m, n, kd):
    rng = np.random.default_rng(m + n + kd)
    A = rng.standard_normal((m, kd)).astype(np.float32)
    B = rng.standard_normal((n, kd)).astype(np.float32)
    C = cat.cat_gemm_f32(torch.from_numpy(A).to(DEV), torch.from_numpy(B).to(DEV)).cpu().numpy()
    ref = A.astype(np.float64) @ B.astype(np.float64).T
    assert np.max(np.abs(C - ref)) <= 1e-5 * np.sqrt(kd) * np.max(np.abs(ref)) + 1e-6
