"""The E4M3 code table of the int4 operand conversion, checked on the CPU against the format.

csrc/int4.cu turns each signed 4-bit value into the byte of an E4M3 number (sign bit, 4-bit
exponent with bias 7, 3-bit fraction) through four 32-bit constants used as byte-permute tables.
Here every byte of those constants is decoded from the format's definition and must equal the
integer it stands for; the GPU parity tests then check the whole GEMM.
"""
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "paper_2302_07594_gb300", "csrc", "int4.cu")


def decode_e4m3(c: int) -> float:
    sign = -1.0 if c & 0x80 else 1.0
    e, f = (c >> 3) & 0xF, c & 0x7
    if e == 0:
        return sign * (f / 8.0) * 2.0 ** -6          # subnormal
    if e == 0xF and f == 0x7:
        return float("nan")                           # the format's only NaN pattern per sign
    return sign * 2.0 ** (e - 7) * (1.0 + f / 8.0)


def table():
    text = open(SRC).read()
    vals = dict(re.findall(r"(kPos0|kPos1|kNeg0|kNeg1) = (0x[0-9A-Fa-f]+)u", text))
    assert set(vals) == {"kPos0", "kPos1", "kNeg0", "kNeg1"}, vals
    words = [int(vals[n], 16) for n in ("kPos0", "kPos1", "kNeg0", "kNeg1")]
    return [(w >> (8 * i)) & 0xFF for w in words for i in range(4)]


def test_codes_decode_to_the_nibble_values():
    codes = table()
    # byte i of (kPos0, kPos1) encodes nibble i (value i); byte i of (kNeg0, kNeg1) nibble 8 + i (value i - 8)
    for nib in range(16):
        value = nib - 16 if nib >= 8 else nib
        assert decode_e4m3(codes[nib]) == value, (nib, hex(codes[nib]))


def test_codes_are_the_unique_encodings():
    # every finite E4M3 value has one code, except zero (0x00 and 0x80): the table uses +0
    codes = table()
    assert codes[0] == 0x00
    for nib in range(1, 16):
        value = nib - 16 if nib >= 8 else nib
        assert [c for c in range(256) if decode_e4m3(c) == value] == [codes[nib]]
