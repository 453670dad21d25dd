"""Full-size parity: the five layer configurations run through the same C-ABI calls that
bench.py times, compared with the oracle on sampled tokens and output channels (which it
computes one by one), and -- where the oracle finishes in seconds -- on the whole output.

Tolerances as in test_gpu_parity.py.  The whole-output oracle check covers the QKV, down and
decode layers.  On every layer, the 70B gate/up layer included, the whole output is also checked by
a property that holds at any size: the same codes and steps through the independent digit-plane
GEMM give the packed GEMM's y bit for bit (both accumulate exactly).  For n > 32 the byte-code calls
that bench.py times for prefill (transform with byte codes out, GEMM with SQNR sums) give the same
codes, steps and y."""
import numpy as np
import pytest
import torch

import dp_planes
import oracle as O
import sm4x8
import workloads as WL
from test_gpu_parity import DEV, check_codes, gpu_layer, rel_fro, to_dev

pytestmark = pytest.mark.gpu

cat = pytest.importorskip("paper_2603_04359_gb300")

FULL_OUTPUT = {"c2_qkv_4096x6144_k128_bf16", "c3_down_14336x4096_k128_bf16", "c4_decode_up_4096x14336_k128_bf16"}


def _y_ref(L):
    torch.backends.cuda.matmul.allow_tf32 = False
    x = torch.from_numpy(L.x_eval.values).to(DEV)
    W = torch.from_numpy(L.W.values).to(DEV)
    return (x @ W.t()).contiguous()


def _planes_on_device(packed: torch.Tensor) -> torch.Tensor:
    """SM4x8 codes [R][d/2] -> one E4M3 digit plane [1][R][d], on the device, from the format's
    definition in the header: the E4M3 bytes of codes e0..e3 of a word w are w & 0x87878787 and those
    of e4..e7 are rotr(w, 4) & 0x87878787, and a code's E4M3 byte is also its one-digit plane byte."""
    R, half = packed.shape
    w = packed.contiguous().view(torch.int32).to(torch.int64) & 0xFFFFFFFF          # [R][d/8] words
    lo = w & 0x87878787
    hi = (((w >> 4) | (w << 28)) & 0xFFFFFFFF) & 0x87878787
    parts = [(lo >> (8 * i)) & 0xFF for i in range(4)] + [(hi >> (8 * i)) & 0xFF for i in range(4)]
    return torch.stack(parts, dim=-1).reshape(1, R, 2 * half).to(torch.uint8)


@pytest.mark.parametrize("name,k,kind", [("c1_256x256_k32_f32", 32, "cat"), ("c2_qkv_4096x6144_k128_bf16", 128, "cat"),
                                         ("c2_qkv_4096x6144_k128_bf16", 128, "identity"),
                                         ("c2_qkv_4096x6144_k128_bf16", 128, "rht"),
                                         ("c3_down_14336x4096_k128_bf16", 128, "cat"),
                                         ("c3_down_14336x4096_k128_bf16", 128, "rht"),
                                         ("c4_decode_up_4096x14336_k128_bf16", 128, "cat"),
                                         ("c5_gateup_8192x28672_bf16", 32, "cat"), ("c5_gateup_8192x28672_bf16", 64, "cat"),
                                         ("c5_gateup_8192x28672_bf16", 128, "cat"),
                                         ("c5_gateup_8192x28672_bf16", 128, "identity"),
                                         ("c5_gateup_8192x28672_bf16", 128, "rht"), ("c5_gateup_8192x28672_bf16", 256, "cat")])
def test_full_size_layer(name, k, kind):
    cfg = WL.CONFIGS[name]
    L = WL.make_layer(cfg)
    n, d_in, d_out = cfg.n_eval, cfg.d_in, cfg.d_out
    g = gpu_layer(L, kind, k)
    assert cat.cat_device_status()[0] == 0

    # oracle: transform from the same calibration split
    Wv = L.W.values
    Sx = Sw = None
    if kind == "cat":
        Xc = L.x_calib.values.astype(np.float64)
        Sx = O.calib_cov_block_sums(Xc, k) / cfg.n_calib
        assert rel_fro(g["sigma"].cpu().numpy(), Sx * cfg.n_calib) < (1e-10 if cfg.dtype == "f32" else 1e-6)
        Sw = O.weight_autocorr_blocks(Wv, k)
    T, Ti = O.build_transform(kind, d_in, k, Sx, Sw, L.rht_signs)
    assert rel_fro(g["T"].cpu().numpy(), T) < (1e-6 if cfg.dtype == "f32" else 1e-5)

    # sampled rows and tokens, computed one by one
    rng = np.random.default_rng(1234)
    ts = np.sort(rng.choice(n, min(n, 48), replace=False))
    os_ = np.sort(rng.choice(d_out, min(d_out, 256), replace=False))
    qw, sw, pre_w = O.quantize_rows_symmetric(O.apply_weight_transform(Wv[os_], Ti))
    qx, sx, pre_x = O.quantize_rows_symmetric(O.apply_act_transform(L.x_eval.values[ts], T))
    qw_g = sm4x8.unpack(g["Wq"][torch.from_numpy(os_).to(DEV)].cpu().numpy())
    qx_g = sm4x8.unpack(g["xq"][torch.from_numpy(ts).to(DEV)].cpu().numpy())
    flips = check_codes(qw_g, qw, pre_w) + check_codes(qx_g, qx, pre_x)
    np.testing.assert_allclose(g["sw"].cpu().numpy()[os_], sw, rtol=1e-5)
    np.testing.assert_allclose(g["sx"].cpu().numpy()[ts], sx, rtol=1e-5)
    y_gpu = g["y"]
    y_gpu_s = y_gpu[torch.from_numpy(ts).to(DEV)][:, torch.from_numpy(os_).to(DEV)].cpu().numpy()
    # given the codes (the oracle's, with the near-boundary differences check_codes accepted), the
    # output is the exact integer product times the oracle's steps
    y_hat_g = O.dequantize_output(O.int_gemm(qx_g, qw_g), sx, sw)
    assert rel_fro(y_gpu_s, y_hat_g) < 1e-5
    y_s = O.linear(L.x_eval.values[ts], Wv[os_])
    assert abs(O.sqnr_db(y_s, y_gpu_s) - O.sqnr_db(y_s, y_hat_g)) < 0.01
    if flips == 0:   # one accepted flip in a heavy-tailed token moves a 48-token sample by ~1e-3
        y_hat_s = O.dequantize_output(O.int_gemm(qx, qw), sx, sw)
        assert rel_fro(y_gpu_s, y_hat_s) < 1e-3

    # whole-output SQNR through cat_sqnr (y_ref from an fp32 GEMM, as bench.py supplies it)
    y_ref = _y_ref(L)
    s3 = cat.cat_sqnr(y_ref, y_gpu).cpu().numpy()
    d = (y_ref.double() - y_gpu.double())
    assert abs(s3[1] - float((d * d).sum())) <= 1e-6 * s3[1]
    # the whole output, at any size: the independent digit-plane GEMM on the same codes and steps
    xp = _planes_on_device(g["xq"])
    ts_d = torch.from_numpy(ts).to(DEV)
    np.testing.assert_array_equal(dp_planes.decode(xp[:, ts_d].cpu().numpy()), sm4x8.unpack(g["xq"][ts_d].cpu().numpy()))
    y_dp = cat.cat_linear_dp(xp, 4, g["sx"], _planes_on_device(g["Wq"]), 4, g["sw"])
    assert torch.equal(y_dp, y_gpu)
    if n > 32:
        # the byte-code calls bench.py times for prefill: the same codes (as bytes, against the format's
        # definition above), the same steps, y bit for bit, the same SQNR sums
        planes = (cat.cat_split_transform(g["T"], k)
                  if (cfg.dtype == "bf16" and cat.cat_split_transform_bytes(d_in, k) > 0) else None)
        xq8, sx8 = cat.cat_transform_quantize_act_e8(to_dev(L.x_eval), g["T"], planes, k)
        assert torch.equal(xq8, xp[0]) and torch.equal(sx8, g["sx"])
        y8, o3 = cat.cat_w4a4_linear_sqnr_e8(xq8, sx8, cat.cat_codes_to_e4m3(g["Wq"]), g["sw"], y_ref)
        assert torch.equal(y8, y_gpu)
        o3 = o3.cpu().numpy()
        assert abs(o3[1] - s3[1]) <= 1e-6 * s3[1] and abs(o3[2] - s3[2]) < 1e-4
        del xq8, y8
    if name in FULL_OUTPUT and kind == "cat":
        ref = O.transform_quantize_act(L.x_eval.values, T)
        prep_q, prep_s, _ = O.quantize_rows_symmetric(O.apply_weight_transform(Wv, Ti))
        _, y_hat = O.w4a4_linear(ref.qx, ref.sx, prep_q, prep_s)
        y = O.linear(L.x_eval.values, Wv)
        assert rel_fro(y_gpu.cpu().numpy(), y_hat) < 1e-3
        assert abs(s3[2] - O.sqnr_db(y, y_hat)) < 0.01
