"""Write fill_tables.h: the constant tables of the 16-bit and 8-bit NORMAL
fill, each entry the correctly rounded fp32 value of its closed form,
computed with 50-digit arithmetic (mpmath).

  angle  (sin, cos) of 2 pi (j + 1/2) / 256, j = 0..255
  rad16  per cell c = 16 E + i (E = 0..31, i = 0..15), with d = [E >= 16],
         e = E - 16 d, m0 = 1 + i/16, g(m) = sqrt(-2 ln y(m)),
         y(m) = m 2^(e-17) (d = 0) or 1 - m 2^(e-17) (d = 1), and the chord
         slope S = 16 (g(m0 + 1/16) - g(m0)):
           A'_c = RN32(S 2^(16-E)),  B_c = RN32(g(m0) - S m0)
         The kernel multiplies A'_c by F 2^-16 (the radius argument F of the
         chord scaled by 2^-16), so A'_c is the chord slope per unit of F
         times 2^16: the product, and so every rho, is the same.
  rad8   sqrt(-2 ln((k + 1/2) / 256)), k = 0..255
  c16    2 pi / 65536

Run:  python gen_fill_tables.py > fill_tables.h
"""
import struct
import sys

import mpmath

mpmath.mp.dps = 50


def rn32(x):
    """The fp32 nearest to x (ties to even)."""
    f = struct.unpack("<f", struct.pack("<f", float(x)))[0]
    bits = struct.unpack("<I", struct.pack("<f", f))[0]
    best = None
    for b in (bits - 1, bits, bits + 1):
        c = struct.unpack("<f", struct.pack("<I", b & 0xFFFFFFFF))[0]
        d = abs(mpmath.mpf(c) - x)
        if best is None or d < best[0] or (d == best[0] and b % 2 == 0):
            best = (d, c)
    return best[1]


def lit(v):
    return "%sf" % float.hex(v) if v >= 0 else "(%sf)" % float.hex(v)


def main(out):
    half = mpmath.mpf(1) / 2
    w = out.write
    w("// fill_tables.h -- constant tables of the 16-bit and 8-bit NORMAL fill.\n")
    w("// Written by gen_fill_tables.py (50-digit arithmetic); every entry is the\n")
    w("// correctly rounded fp32 value of the closed form stated there.\n")
    w("#pragma once\n\n")
    w("// (sin, cos) of 2 pi (j + 1/2) / 256\n")
    w("static __device__ const float2 kAngleTable[256] = {\n")
    for j in range(256):
        phi = 2 * mpmath.pi * (j + half) / 256
        w("    {%s, %s},\n" % (lit(rn32(mpmath.sin(phi))), lit(rn32(mpmath.cos(phi)))))
    w("};\n\n")
    w("// 16-bit radius chords: rho = fma(F 2^-16, A'_c, B_c), entry c = (A'_c, B_c)\n")
    w("static __device__ const float2 kRadius16Table[512] = {\n")
    for E in range(32):
        d = 1 if E >= 16 else 0
        e = E - 16 * d
        for i in range(16):
            m0 = 1 + mpmath.mpf(i) / 16
            m1 = m0 + mpmath.mpf(1) / 16

            def g(m):
                y = m * mpmath.mpf(2) ** (e - 17)
                return mpmath.sqrt(-2 * mpmath.log(1 - y if d else y))
            S = 16 * (g(m1) - g(m0))
            w("    {%s, %s},\n" % (lit(rn32(S * mpmath.mpf(2) ** (16 - E))), lit(rn32(g(m0) - S * m0))))
    w("};\n\n")
    w("// 8-bit radii sqrt(-2 ln((k + 1/2) / 256))\n")
    w("static __device__ const float kRadius8Table[256] = {\n")
    for k in range(256):
        w("    %s,\n" % lit(rn32(mpmath.sqrt(-2 * mpmath.log((k + half) / 256)))))
    w("};\n\n")
    c16 = rn32(2 * mpmath.pi / 65536)
    w("#define ASMV_C16 %s          /* 2 pi / 65536 */\n" % lit(c16))
    w("#define ASMV_C16_HALF %s     /* its half (exact) */\n" % lit(c16 / 2))


if __name__ == "__main__":
    main(sys.stdout)
