"""Byte codes (one E4M3 byte per INT4 code) and the GEMM that reads them without a decode step,
through the C ABI: the conversion is bit-exact against the byte encoding written out here, the
accumulators match the oracle's integer GEMM bit for bit, and y and the SQNR sums are identical to
the SM4x8 GEMM's (same exact accumulators, same scaling)."""
import numpy as np
import pytest
import torch

import oracle as O
import sm4x8
import workloads as WL

pytestmark = pytest.mark.gpu

cat = pytest.importorskip("paper_2603_04359_gb300")
DEV = "cuda"


def byte_codes(q: np.ndarray) -> np.ndarray:
    """The E4M3 byte of the subnormal q * 2^-9: sign bit 7, magnitude in bits 0-2."""
    q = np.asarray(q, dtype=np.int64)
    return (np.where(q < 0, 0x80, 0) | np.abs(q)).astype(np.uint8)


def rel_fro(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("rows,d", [(1, 32), (77, 4096), (1000, 160), (3, 262144)])
def test_codes_to_e4m3(rows, d):
    rng = np.random.default_rng(rows + d)
    q = WL.random_codes(rng, (rows, d)).astype(np.int64)
    q[0, :15] = np.arange(-7, 8)                           # every code value
    out = cat.cat_codes_to_e4m3(torch.from_numpy(sm4x8.pack(q)).to(DEV))
    np.testing.assert_array_equal(out.cpu().numpy(), byte_codes(q))


E8_SHAPES = [
    (1, 64, 8), (17, 96, 33), (32, 384, 300),            # n <= 32: one partly filled 256-row tile
    (33, 128, 256), (128, 256, 256), (129, 160, 300), (300, 384, 520), (257, 4096, 64),
    (512, 1024, 1024), (1024, 512, 6144),                # several tiles per pair
    (256, 1024, 9984), (300, 2048, 5030),                # a last wave split along K into 4 / 8 parts
    # 256-channel pair tiles (chosen where they take less time on 76 pairs), ragged rows and columns
    (2048, 4096, 6144), (4096, 512, 6144), (2000, 1024, 10000), (600, 2048, 30000),
]


@pytest.mark.parametrize("n,d_in,d_out", E8_SHAPES)
def test_w4a4_linear_e8_exact(n, d_in, d_out):
    rng = np.random.default_rng(n * 1000 + d_in + d_out)
    qx = WL.random_codes(rng, (n, d_in)).astype(np.int64)
    qw = WL.random_codes(rng, (d_out, d_in)).astype(np.int64)
    sx = rng.uniform(0.01, 2.0, n).astype(np.float32)
    sw = rng.uniform(0.001, 0.1, d_out).astype(np.float32)
    sx_d, sw_d = torch.from_numpy(sx).to(DEV), torch.from_numpy(sw).to(DEV)
    xq8 = torch.from_numpy(byte_codes(qx)).to(DEV)
    wq8 = cat.cat_codes_to_e4m3(torch.from_numpy(sm4x8.pack(qw)).to(DEV))   # the weights' preparation
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    y = cat.cat_w4a4_linear_e8(xq8, sx_d, wq8, sw_d, acc_out=acc)
    ref_acc = O.int_gemm(qx, qw)
    np.testing.assert_array_equal(acc.cpu().numpy(), ref_acc)
    ref_y = O.dequantize_output(ref_acc, sx.astype(np.float64), sw.astype(np.float64))
    assert rel_fro(y.cpu().numpy(), ref_y) < 1e-6
    if n > 32:                                          # the SM4x8 tile GEMM: the same y, bit for bit
        y4 = cat.cat_w4a4_linear(torch.from_numpy(sm4x8.pack(qx)).to(DEV), sx_d,
                                 torch.from_numpy(sm4x8.pack(qw)).to(DEV), sw_d)
        assert torch.equal(y, y4)
    assert cat.cat_device_status()[0] == 0


@pytest.mark.parametrize("n,d_in", [(200, 14336), (40, 4096)])
def test_w4a4_linear_e8_extreme_accumulators(n, d_in):
    d_out = 64
    qx = np.full((n, d_in), 7, dtype=np.int64)
    qx[1::2] = -7
    qw = np.full((d_out, d_in), 7, dtype=np.int64)
    qw[3, : d_in // 2] = -7                       # cancels to zero
    qw[5, -300:] = np.arange(300) % 3 - 1         # small codes after a large prefix
    ones = torch.ones(max(n, d_out), dtype=torch.float32, device=DEV)
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    cat.cat_w4a4_linear_e8(torch.from_numpy(byte_codes(qx)).to(DEV), ones[:n].contiguous(),
                           torch.from_numpy(byte_codes(qw)).to(DEV), ones[:d_out].contiguous(), acc_out=acc)
    ref = O.int_gemm(qx, qw)
    assert np.abs(ref).max() == 49 * d_in
    np.testing.assert_array_equal(acc.cpu().numpy(), ref)


@pytest.mark.parametrize("n,d_in,d_out", [(300, 1024, 520), (513, 512, 256), (257, 4096, 130), (16, 1024, 200),
                                          (1024, 512, 6144), (300, 2048, 5032),
                                          (2000, 1024, 10000), (4096, 512, 6144)])   # 256-channel tiles
def test_w4a4_linear_sqnr_e8(n, d_in, d_out):
    """y equals cat_w4a4_linear_e8's bit for bit; the sums match the oracle's over the same outputs and,
    for n > 32, the SM4x8 call's (to the sums' precision: the tiles may group the outputs differently)."""
    rng = np.random.default_rng(n + 7 * d_in + 13 * d_out)
    qx = WL.random_codes(rng, (n, d_in)).astype(np.int64)
    qw = WL.random_codes(rng, (d_out, d_in)).astype(np.int64)
    sx = rng.uniform(0.01, 2.0, n).astype(np.float32)
    sw = rng.uniform(0.001, 0.1, d_out).astype(np.float32)
    sx_d, sw_d = torch.from_numpy(sx).to(DEV), torch.from_numpy(sw).to(DEV)
    xq8, wq8 = torch.from_numpy(byte_codes(qx)).to(DEV), torch.from_numpy(byte_codes(qw)).to(DEV)
    y_plain = cat.cat_w4a4_linear_e8(xq8, sx_d, wq8, sw_d)
    y_ref = (y_plain.double() + torch.randn(n, d_out, device=DEV, dtype=torch.float64) * 0.05).float().contiguous()
    for rep in range(2):                                   # twice: the sums restart from zero each call
        y, out3 = cat.cat_w4a4_linear_sqnr_e8(xq8, sx_d, wq8, sw_d, y_ref)
        assert torch.equal(y, y_plain)
        sig, err = O.sqnr_sums(y_ref.cpu().numpy(), y.cpu().numpy())
        o = out3.cpu().numpy()
        assert abs(o[0] - sig) <= 1e-6 * sig and abs(o[1] - err) <= 1e-6 * err
        assert abs(o[2] - 10 * np.log10(sig / err)) < 1e-5
    if n > 32:
        # the same outputs; the sums may group them differently (256-channel tiles): fp32 runs, ~1e-10
        _, out4 = cat.cat_w4a4_linear_sqnr(torch.from_numpy(sm4x8.pack(qx)).to(DEV), sx_d,
                                           torch.from_numpy(sm4x8.pack(qw)).to(DEV), sw_d, y_ref)
        torch.testing.assert_close(out3, out4, rtol=1e-9, atol=0)
    assert cat.cat_device_status()[0] == 0


# ------------------------------------------------------------------------------------------
# cat_transform_quantize_act_e8: the same code decisions, written as byte codes
# ------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,d,k,dtype", [(67, 384, 128, "bf16"), (1000, 256, 128, "bf16"),      # fused, one wave
                                         (2560, 4096, 128, "bf16"), (1300, 8192, 64, "bf16"),   # fused in waves
                                         (300, 512, 32, "bf16"), (300, 192, 64, "bf16"),        # embedded, 64-wide
                                         (2560, 4096, 256, "bf16"), (200, 512, 256, "bf16"),    # k = 256 quarters
                                         (1100, 9920, 64, "bf16"), (520, 20480, 128, "bf16"),   # two passes + convert
                                         (1300, 10240, 256, "bf16"),                             # SIMT + convert
                                         (130, 256, 32, "f32"), (5, 64, 16, "bf16")])            # SIMT + convert
def test_transform_quantize_act_e8(n, d, k, dtype):
    """The byte codes are the byte form of cat_transform_quantize_act_split's SM4x8 codes and the steps
    are the same, bit for bit; on the first shape also checked against the oracle directly."""
    from test_gpu_parity import _cat_T, check_codes, to_dev
    rng = np.random.default_rng(11 * n + d)
    X = rng.standard_normal((n, d)) * rng.lognormal(0, 1.0, d)
    X[0] = 0.0                       # all-zero token
    X[min(2, n - 1)] *= 1e4          # a huge token
    Xt = WL.cast(X, dtype)
    T32 = _cat_T(rng, d, k)
    Td = torch.from_numpy(T32).to(DEV)
    planes = cat.cat_split_transform(Td, k) if (dtype == "bf16" and cat.cat_split_transform_bytes(d, k) > 0) else None
    xq, sx = cat.cat_transform_quantize_act_split(to_dev(Xt), Td, planes, k)
    xq8, sx8 = cat.cat_transform_quantize_act_e8(to_dev(Xt), Td, planes, k)
    q = sm4x8.unpack(xq.cpu().numpy())
    np.testing.assert_array_equal(xq8.cpu().numpy(), byte_codes(q))
    assert torch.equal(sx, sx8)
    if (n, d, k) == (67, 384, 128):
        ref = O.transform_quantize_act(Xt.values, T32.astype(np.float64))
        b = xq8.cpu().numpy().astype(np.int64)
        check_codes(np.where(b & 0x80, -(b & 0x7F), b & 0x7F), ref.qx, ref.pre_x)
    assert cat.cat_device_status()[0] == 0
