"""Independent reader/writer of the library's digit-plane code format (test helper).

Decoding goes through the FP8 E4M3 *value* of each byte (sign, 4-bit exponent with bias 7, 3-bit
mantissa, subnormals below exponent 1), so a test also checks that the library's bytes are the digit
values d * 2^-9 the format promises."""
import numpy as np


def e4m3_value(b: np.ndarray) -> np.ndarray:
    b = np.asarray(b, dtype=np.int64)
    s = np.where(b >> 7, -1.0, 1.0)
    e = (b >> 3) & 0xF
    m = b & 7
    val = np.where(e == 0, m / 8.0 * 2.0 ** -6, (1 + m / 8.0) * 2.0 ** (e.astype(np.float64) - 7))
    return s * val


def decode(planes: np.ndarray) -> np.ndarray:
    """[D][R][d] bytes -> int64 codes sum_p 16^p d_p, with d_p = E4M3 value * 2^9."""
    planes = np.asarray(planes)
    d = e4m3_value(planes) * 512.0
    assert np.all(d == np.rint(d)), "a byte is not an integer digit times 2^-9"
    d = np.rint(d).astype(np.int64)
    return sum(d[p] * 16 ** p for p in range(planes.shape[0]))


def _byte(d: np.ndarray) -> np.ndarray:
    return (np.where(d < 0, 0x80, 0) | np.abs(d)).astype(np.uint8)


def encode(q: np.ndarray, bits: int, asym: bool) -> np.ndarray:
    """int codes -> [D][R][d] digit bytes, per the header's format."""
    q = np.asarray(q, dtype=np.int64)
    if bits <= 4:
        return _byte(q)[None]
    if asym:
        return np.stack([_byte(q & 15), _byte(q >> 4)])
    d0 = ((q + 8) & 15) - 8
    return np.stack([_byte(d0), _byte((q - d0) // 16)])
