"""float32 natural logarithm from a published series (oracle side).

Method (the classical argument reduction of Cody & Waite, "Software Manual for
the Elementary Functions", 1980, with the atanh series):
  x = m * 2^e with m in [sqrt(1/2), sqrt(2)]
  ln m = 2 atanh(s), s = (m - 1) / (m + 1), |s| <= 0.1716
       = 2 s + s * z * (2/3 + z (2/5 + z (2/7 + z (2/9 + z (2/11 + z 2/13))))),  z = s^2
  ln x = e * ln2_hi + (e * ln2_lo + ln m)
Truncation error of the series is below 1e-12; the result is within a few
float32 ulps of ln x.  Every step is a single correctly rounded float32
operation in a fixed order (no fused multiply-add), so any IEEE-754 machine
evaluating the same sequence gets the same bits.

Valid for positive, finite, normal float32 inputs (the sampler only calls it on
values in [2^-24, 17)).  Pinned against math.log in tests/test_oracle_sampler.py.
"""
import numpy as np

F = np.float32
LN2_HI = F(float.fromhex("0x1.62e4p-1"))        # 0.693145751953125, 9 trailing zero bits
LN2_LO = F(float.fromhex("0x1.7f7d1cp-20"))     # float32(ln 2 - LN2_HI)
C = [F(2) / F(2 * k + 1) for k in range(1, 7)]  # 2/3, 2/5, ..., 2/13 (correctly rounded)
SQRT2_BITS = np.uint32(0x3FB504F3)


def flog(x) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    bits = x.view(np.uint32)
    e = (bits >> np.uint32(23)).astype(np.int32) - 127
    mbits = (bits & np.uint32(0x7FFFFF)) | np.uint32(0x3F800000)
    big = mbits > SQRT2_BITS
    m = mbits.view(np.float32)
    m = np.where(big, m * F(0.5), m).astype(np.float32)
    e = e + big.astype(np.int32)
    s = (m - F(1)) / (m + F(1))
    z = s * s
    p = C[5]
    p = C[4] + z * p
    p = C[3] + z * p
    p = C[2] + z * p
    p = C[1] + z * p
    p = C[0] + z * p
    r = z * p
    lnm = (s + s) + s * r
    ef = e.astype(np.float32)
    return (ef * LN2_HI + (ef * LN2_LO + lnm)).astype(np.float32)
