"""Host-side reader/writer of the SM4x8 INT4 code format documented in include/cat_w4a4.h.

Test helper only: it packs oracle codes for GEMM inputs and unpacks the library's codes for
comparison.  Layout: 8 consecutive codes e0..e7 of a row share one little-endian 32-bit word;
byte i holds |e_i| in bits 0-2, sign(e_i) in bit 7, |e_{4+i}| in bits 4-6 and sign(e_{4+(i+3)%4})
in bit 3.
"""
import numpy as np


def pack(q: np.ndarray) -> np.ndarray:
    q = np.asarray(q, dtype=np.int64)
    rows, d = q.shape
    assert d % 8 == 0 and np.all(np.abs(q) <= 7)
    g = q.reshape(rows, d // 8, 8)
    mag = np.abs(g).astype(np.uint8)
    sgn = (g < 0).astype(np.uint8)
    out = np.zeros((rows, d // 8, 4), dtype=np.uint8)
    for i in range(4):
        out[:, :, i] = (mag[:, :, i] | (sgn[:, :, 4 + (i + 3) % 4] << 3) | (mag[:, :, 4 + i] << 4)
                        | (sgn[:, :, i] << 7))
    return out.reshape(rows, d // 2)


def unpack(b: np.ndarray) -> np.ndarray:
    b = np.asarray(b, dtype=np.uint8)
    rows, half = b.shape
    w = b.reshape(rows, half // 4, 4).astype(np.int64)
    out = np.zeros((rows, half // 4, 8), dtype=np.int64)
    for i in range(4):
        m_lo, s_lo = w[:, :, i] & 7, (w[:, :, i] >> 7) & 1
        m_hi, s_hi = (w[:, :, i] >> 4) & 7, (w[:, :, (i + 1) % 4] >> 3) & 1
        out[:, :, i] = np.where(s_lo == 1, -m_lo, m_lo)
        out[:, :, 4 + i] = np.where(s_hi == 1, -m_hi, m_hi)
    return out.reshape(rows, half * 2)


def e4m3_value(byte: np.ndarray) -> np.ndarray:
    """Value of an FP8 E4M3 byte (OCP: bias 7, subnormals 2^-6 * m/8); NaN pattern not used here."""
    byte = np.asarray(byte, dtype=np.int64)
    s = np.where((byte >> 7) & 1, -1.0, 1.0)
    e = (byte >> 3) & 15
    m = byte & 7
    return s * np.where(e == 0, m / 8.0 * 2.0 ** -6, (1 + m / 8.0) * 2.0 ** (e - 7))
