"""cat_quantize_weights_noalloc: weight preparation from the library's static device scratch.

Collected last on purpose: it must give the same results as cat_quantize_weights when run alone
and after every other test (the scratch persists on the device between calls).  Tolerances are
those of the parity tests: transform blocks 1e-6 relative Frobenius, codes +-1 in at most 1e-4 of
the elements (at least one), steps 1e-5 relative."""
import ctypes

import numpy as np
import pytest
import torch

import sm4x8
import workloads as WL

cat = pytest.importorskip("paper_2603_04359_gb300")
DEV = "cuda"

LAYERS = [  # two different shapes and dtypes, prepared back to back through the same scratch
    WL.small_config("nz_bf16_k128", d_in=1024, d_out=640, n_eval=64, n_calib=512, k=128, seed=31),
    WL.small_config("nz_f32_k32", d_in=544, d_out=300, n_eval=64, n_calib=256, k=32, dtype="f32",
                    act="wishart_outlier", seed=32),
]


def _to_dev(t: WL.Tensor) -> torch.Tensor:
    if t.dtype == "f32":
        return torch.from_numpy(np.ascontiguousarray(t.raw)).to(DEV)
    return torch.from_numpy(np.ascontiguousarray(t.raw).view(np.int16)).view(torch.bfloat16).to(DEV)


def _rel_fro(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _compare(got, ref):
    T, Wq, sw = (t.cpu() for t in got)
    Tr, Wqr, swr = (t.cpu() for t in ref)
    assert _rel_fro(T.numpy().astype(np.float64), Tr.numpy().astype(np.float64)) <= 1e-6
    np.testing.assert_allclose(sw.numpy(), swr.numpy(), rtol=1e-5, atol=0)
    qa, qb = sm4x8.unpack(Wq.numpy()).astype(np.int64), sm4x8.unpack(Wqr.numpy()).astype(np.int64)
    diff = qa != qb
    assert np.all(np.abs(qa - qb) <= 1)
    assert diff.sum() <= max(1, int(1e-4 * diff.size))


class _DefaultPool:
    """Used-memory high watermark of the device's default stream-ordered pool (driver API)."""

    USED_MEM_HIGH = 8  # CU_MEMPOOL_ATTR_USED_MEM_HIGH

    def __init__(self, ordinal: int):
        self.ok = False
        try:
            self.cu = ctypes.CDLL("libcuda.so.1")
            dev = ctypes.c_int(0)
            self.pool = ctypes.c_void_p(0)
            self.ok = (self.cu.cuDeviceGet(ctypes.byref(dev), ordinal) == 0 and
                       self.cu.cuDeviceGetDefaultMemPool(ctypes.byref(self.pool), dev) == 0)
        except OSError:
            self.ok = False

    def reset(self) -> bool:
        zero = ctypes.c_uint64(0)
        return self.ok and self.cu.cuMemPoolSetAttribute(self.pool, self.USED_MEM_HIGH, ctypes.byref(zero)) == 0

    def high(self):
        v = ctypes.c_uint64(0)
        if not self.ok or self.cu.cuMemPoolGetAttribute(self.pool, self.USED_MEM_HIGH, ctypes.byref(v)) != 0:
            return None
        return int(v.value)


@pytest.mark.gpu
def test_noalloc_matches_quantize_weights_on_consecutive_calls():
    pool = _DefaultPool(torch.cuda.current_device())
    if not pool.ok:
        pytest.fail("the default stream-ordered pool could not be opened through libcuda: the no-allocation "
                    "check would not run")
    for i, cfg in enumerate(LAYERS):
        L = WL.make_layer(cfg)
        k = cfg.k
        W, xc = _to_dev(L.W), _to_dev(L.x_calib)
        sig = cat.cat_calib_cov(xc, k)
        torch.cuda.synchronize()
        # control: the allocating entry point raises the pool's high watermark, so the watch works
        assert pool.reset()
        ref = cat.cat_quantize_weights(W, k, "cat", sigma_x=sig, n_calib=cfg.n_calib)
        torch.cuda.synchronize()
        control = pool.high()
        if not control:
            pytest.fail(f"the allocating entry point left the pool's watermark at {control}: the watch cannot "
                        "tell an allocation from none")
        # preallocated outputs, so that nothing but the call itself runs between the two readings
        out = (torch.full_like(ref[0], float("nan")), torch.full_like(ref[1], 0xFF), torch.full_like(ref[2], -1.0))
        torch.cuda.synchronize()
        assert pool.reset()
        free_before = torch.cuda.mem_get_info()[0]
        got = cat.cat_quantize_weights_noalloc(W, k, "cat", sigma_x=sig, n_calib=cfg.n_calib, out=out)
        torch.cuda.synchronize()
        free_after = torch.cuda.mem_get_info()[0]
        assert pool.high() == 0, "the no-alloc entry point took memory from the stream-ordered pool"
        if i > 0:
            # after the first call (which may load the library's modules and their static scratch onto
            # the device) no call takes device memory of any kind
            assert free_after == free_before, f"free device memory moved by {free_before - free_after} bytes"
        assert cat.cat_device_status()[0] == 0
        _compare(got, ref)


@pytest.mark.gpu
def test_noalloc_identity_and_rht_match():
    cfg = LAYERS[0]
    L = WL.make_layer(cfg)
    W = _to_dev(L.W)
    for kind in ("identity", "rht"):
        signs = L.rht_signs if kind == "rht" else None
        ref = cat.cat_quantize_weights(W, cfg.k, kind, rht_signs=signs)
        got = cat.cat_quantize_weights_noalloc(W, cfg.k, kind, rht_signs=signs)
        _compare(got, ref)


def test_noalloc_rejects_sizes_beyond_the_scratch():
    """d_in * k above the static limit is refused before any CUDA call (runs without a GPU)."""
    lib = cat.load_library()
    P = ctypes.c_void_p(0x10000)
    d_in, k = 16384, 128                                   # d_in * k = 2^21 > 2^20
    st = lib.cat_quantize_weights_noalloc(P, 1, 64, d_in, k, 0, None, 0, None, P, P, P, None)
    assert st == 2                                         # CAT_ERR_SHAPE
    assert b"CAT_PREP_NOALLOC_MAX_DK" in lib.cat_last_error()
    st = lib.cat_quantize_weights_noalloc(P, 1, 64, 4096, 512, 0, None, 0, None, P, P, P, None)
    assert st == 2                                         # k = 512 is not a block size either
