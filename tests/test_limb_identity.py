"""The arithmetic identities the GPU kernels rest on, checked exhaustively on the CPU (no GPU).

These restate, independently of both the oracle and the CUDA sources, the integer facts that make
the tensor-core path exact:

* centred limbs: every int16 a is 256*h + l with h = floor((a + 128) / 256) in [-128, 128] and
  l = a - 256*h in [-128, 127], both exact in fp16, so every limb product is exact in fp32 with
  magnitude <= 2^14;
* the limb product identity 2^16*h_a*h_b + 2^8*(h_a*l_b + l_a*h_b) + l_a*l_b = a*b over all 2^32
  pairs (a, b) of int16 values (a small C program, a few seconds);
* the byte logic with which the fused kernel splits raw int16 pairs on chip: for the two's-complement
  bytes lo, hi of a, l + 128 = lo ^ 0x80 and h + 128 = (hi ^ 0x80) + (lo >> 7);
* the int8 -> fp16 conversion: the fp16 with bit pattern 0x6400 | (v ^ 0x80) is 1024 + v + 128, so
  one subtraction of 1152 gives v exactly, for every int8 v;
* the skinny kernel's non-centred limbs b = 256*(b >> 8) + (b & 255) and its chunk bounds.
"""
import os
import subprocess
import tempfile

import numpy as np

ALL16 = np.arange(-32768, 32768, dtype=np.int64)


def centred(a):
    h = np.floor_divide(a + 128, 256)
    return h, a - 256 * h


def test_centred_limbs_ranges_and_fp16_exactness():
    h, l = centred(ALL16)
    assert np.array_equal(256 * h + l, ALL16)
    assert h.min() == -128 and h.max() == 128
    assert l.min() == -128 and l.max() == 127
    for x in (h, l):
        assert np.array_equal(x.astype(np.float16).astype(np.int64), x)  # exact in fp16
    # the largest limb product magnitude, and fp32 exactness of chunk sums up to 2^24
    assert max(abs(int(h.min())), int(h.max())) ** 2 == 1 << 14
    assert np.float32(1 << 24) - np.float32((1 << 24) - 1) == 1.0


LIMB_PAIRS_C = r"""
#include <stdint.h>
#include <stdio.h>
static int64_t floordiv256(int64_t x) { return x >= 0 ? x / 256 : -((-x + 255) / 256); }
int main(void) {
  uint64_t bad = 0;
  for (int64_t a = -32768; a <= 32767; ++a) {
    const int64_t ha = floordiv256(a + 128), la = a - 256 * ha;
    for (int64_t b = -32768; b <= 32767; ++b) {
      const int64_t hb = floordiv256(b + 128), lb = b - 256 * hb;
      const int64_t v = 65536 * ha * hb + 256 * (ha * lb + la * hb) + la * lb;
      bad += (v != a * b);
    }
  }
  printf("%llu\n", (unsigned long long)bad);
  return bad != 0;
}
"""


def test_limb_product_identity_all_pairs():
    with tempfile.TemporaryDirectory() as d:
        src, exe = os.path.join(d, "limbs.c"), os.path.join(d, "limbs")
        open(src, "w").write(LIMB_PAIRS_C)
        subprocess.run(["gcc", "-O2", "-std=c11", src, "-o", exe], check=True, capture_output=True)
        r = subprocess.run([exe], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and r.stdout.strip() == "0", r.stdout


def test_fused_byte_logic_split():
    u = ALL16 & 0xFFFF
    lo, hi = u & 0xFF, u >> 8
    h, l = centred(ALL16)
    assert np.array_equal(l + 128, lo ^ 0x80)
    assert np.array_equal(h + 128, (hi ^ 0x80) + (lo >> 7))
    # both biased limbs sit under the fp16 exponent of 1024: 0x6400 | x is 1024 + x for x <= 256,
    # and one fp16 subtraction of 1152 = 1024 + 128 recovers the limb exactly
    for x, limb in ((lo ^ 0x80, l), ((hi ^ 0x80) + (lo >> 7), h)):
        assert x.max() <= 256
        f = (np.uint16(0x6400) + x.astype(np.uint16)).view(np.float16)
        assert np.array_equal((f - np.float16(1152)).astype(np.int64), limb)


def test_int8_to_fp16_bit_trick():
    v = np.arange(-128, 128, dtype=np.int64)
    bits = (0x6400 | ((v ^ 0x80) & 0xFF)).astype(np.uint16)
    f = bits.view(np.float16)
    assert np.array_equal(f.astype(np.int64), 1024 + v + 128)
    assert np.array_equal((f - np.float16(1152)).astype(np.int64), v)


def test_skinny_non_centred_limbs_and_chunk_bounds():
    hi, lo = ALL16 >> 8, ALL16 & 255
    assert np.array_equal(256 * hi + lo, ALL16)
    assert hi.min() == -128 and hi.max() == 127 and lo.min() == 0 and lo.max() == 255
    # 128-index chunks: the low-low and the cross sums stay below 2^23
    assert 128 * 255 * 255 < 1 << 23
    assert 128 * 2 * 128 * 255 < 1 << 23
