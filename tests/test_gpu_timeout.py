"""A bounded device wait that runs out: the kernel gives up cleanly and the library recovers.

cat_set_wait_limit_ns shortens the pipeline waits of the weight-streaming GEMM and the digit-plane
GEMM to 1 ns, so the first wait that is not satisfied at once gives up.  No GPU fault is involved:
the kernel drains its copies and MMAs in flight (those waits keep their 1 s bound), frees its
tensor memory and returns; the host reads CAT_ERR_TIMEOUT with the kernel's bit and a source line
from the status word.  The next call at the default bound must then succeed with exact results."""
import numpy as np
import pytest
import torch

import dp_planes
import oracle as O
import sm4x8
import workloads as WL

pytestmark = pytest.mark.gpu

cat = pytest.importorskip("paper_2603_04359_gb300")
DEV = "cuda"
CAT_ERR_TIMEOUT = 7


def _decode_call(rng):
    n, d_in, d_out = 16, 4096, 2048
    qx = WL.random_codes(rng, (n, d_in)).astype(np.int64)
    qw = WL.random_codes(rng, (d_out, d_in)).astype(np.int64)
    xq = torch.from_numpy(sm4x8.pack(qx)).to(DEV)
    wq = torch.from_numpy(sm4x8.pack(qw)).to(DEV)
    ones_x, ones_w = torch.ones(n, device=DEV), torch.ones(d_out, device=DEV)
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    return (lambda: cat.cat_w4a4_linear(xq, ones_x, wq, ones_w, acc_out=acc)), acc, O.int_gemm(qx, qw), 1 << 11


def _dp_call(rng):
    n, d_in, d_out, bits = 256, 4096, 512, 8
    qx = rng.integers(-127, 128, (n, d_in))
    qw = rng.integers(-127, 128, (d_out, d_in))
    xp = torch.from_numpy(dp_planes.encode(qx, bits, False)).to(DEV)
    wp = torch.from_numpy(dp_planes.encode(qw, bits, False)).to(DEV)
    ones_x, ones_w = torch.ones(n, device=DEV), torch.ones(d_out, device=DEV)
    acc = torch.empty((n, d_out), dtype=torch.int32, device=DEV)
    return (lambda: cat.cat_linear_dp(xp, bits, ones_x, wp, bits, ones_w, acc_out=acc)), acc, O.int_gemm(qx, qw), 1 << 13


@pytest.mark.parametrize("make", [_decode_call, _dp_call], ids=["weight_streaming_gemm", "digit_plane_gemm"])
def test_bounded_wait_gives_up_then_library_recovers(make):
    call, acc, ref, kernel_bit = make(np.random.default_rng(17))
    assert cat.cat_device_status()[0] == 0                    # clean start
    try:
        cat.cat_set_wait_limit_ns(1)
        call()
        st, word = cat.cat_device_status()
    finally:
        cat.cat_set_wait_limit_ns(0)                          # back to the default bound (1 s)
    assert st == CAT_ERR_TIMEOUT, (st, hex(word))
    assert word & 1 and word & kernel_bit, hex(word)
    assert (word >> 16) > 0, "the source line of the first wait that gave up"
    # the context is intact: the same call at the default bound is exact, twice
    for _ in range(2):
        acc.fill_(0)
        call()
        assert cat.cat_device_status()[0] == 0
        np.testing.assert_array_equal(acc.cpu().numpy(), ref)
