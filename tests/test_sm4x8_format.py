"""The SM4x8 code format: round trip, and the property the GEMM relies on (two masks turn a
word into the E4M3 bytes of its eight codes, worth q * 2^-9 each)."""
import numpy as np

import sm4x8


def test_roundtrip_all_codes():
    rng = np.random.default_rng(0)
    q = rng.integers(-7, 8, (37, 256))
    q[0, :15] = np.arange(-7, 8)
    np.testing.assert_array_equal(sm4x8.unpack(sm4x8.pack(q)), q)


def test_masks_give_e4m3_of_codes():
    rng = np.random.default_rng(1)
    q = rng.integers(-7, 8, (5, 64))
    words = sm4x8.pack(q).view("<u4").astype(np.uint64)
    lo = words & 0x87878787
    hi = ((words >> 4) | (words << 28)) & 0x87878787  # rotate right by 4 within 32 bits
    for r in range(5):
        for wi in range(8):
            for i in range(4):
                blo = (int(lo[r, wi]) >> (8 * i)) & 0xFF
                bhi = (int(hi[r, wi]) >> (8 * i)) & 0xFF
                assert sm4x8.e4m3_value(blo) == q[r, 8 * wi + i] * 2.0 ** -9
                assert sm4x8.e4m3_value(bhi) == q[r, 8 * wi + 4 + i] * 2.0 ** -9


def test_e4m3_decoder_reference_points():
    # OCP E4M3: 0x38 = 1.0, 0x40 = 2.0, 0x7E = 448, 0x01 = 2^-9 (smallest subnormal), 0x08 = 2^-6
    assert sm4x8.e4m3_value(0x38) == 1.0 and sm4x8.e4m3_value(0x40) == 2.0
    assert sm4x8.e4m3_value(0x7E) == 448.0 and sm4x8.e4m3_value(0xB8) == -1.0
    assert sm4x8.e4m3_value(0x01) == 2.0 ** -9 and sm4x8.e4m3_value(0x08) == 2.0 ** -6


def test_byte_codes_are_the_mask_bytes():
    """Byte codes (one E4M3 byte per code, the byte-code GEMM's operand) are exactly the bytes the
    SM4x8 masks produce: (q < 0) << 7 | |q|, worth q * 2^-9."""
    q = np.tile(np.arange(-7, 8), 8)[:64].reshape(2, 32)
    words = sm4x8.pack(q).view("<u4").astype(np.uint64)
    lo = words & 0x87878787
    hi = ((words >> 4) | (words << 28)) & 0x87878787
    for r in range(2):
        for wi in range(4):
            for i in range(4):
                for b, code in (((int(lo[r, wi]) >> (8 * i)) & 0xFF, q[r, 8 * wi + i]),
                                ((int(hi[r, wi]) >> (8 * i)) & 0xFF, q[r, 8 * wi + 4 + i])):
                    assert b == ((0x80 if code < 0 else 0) | abs(int(code)))
                    assert sm4x8.e4m3_value(b) == code * 2.0 ** -9

