"""Planted mistakes in the oracle must each fail at least one of its pins.

Each mutant below is one plausible slip in oracle/asmv_oracle.c: a dropped
term, a wrong sign, index or operand, a wrong rounding or tie rule, an
off-by-one scale.  The test compiles the edited source with the oracle's
own flags into a temporary library, routes the oracle module to it, and
runs the oracle's pin tests (every test_oracle_* function and every
parametrisation of it) from cheapest to dearest until one fails.  A mutant
that passes every pin would mean the pins do not fix that part of the
oracle, so it fails this test.  All of it runs on the CPU.
"""
import importlib
import itertools
import os

import pytest

from oracle import build as oracle_build
from oracle import oracle as O

PIN_MODULES = ("tests.test_oracle_codecs", "tests.test_oracle_philox",
               "tests.test_oracle_fill", "tests.test_oracle_compare",
               "tests.test_oracle_eq", "tests.test_oracle_dtypes", "tests.test_oracle_restore",
               "tests.test_oracle_boxmuller", "tests.test_oracle_eq64",
               "tests.test_oracle_narrow")
# pins that take seconds run last, in this order
EXPENSIVE = ("test_normal16_is_standard_normal", "test_narrow_tables_are_correctly_rounded",
             "test_boxmuller_is_standard_normal", "test_sincos_2pi_u24_all_inputs",
             "test_ln_u24_all_inputs")

# (name, text in the oracle source, replacement): each text occurs once
MUTANTS = [
    # Philox4x32-10 (Salmon et al., SC'11)
    ("philox_key_bump_dropped", "k0 += PHILOX_W_0; k1 += PHILOX_W_1;", "k0 += PHILOX_W_0;"),
    ("philox_bump_before_first_round", "if (round > 0) {", "if (round >= 0) {"),
    ("philox_xor_wrong_word", "uint32_t y0 = pb_hi ^ x1 ^ k0;", "uint32_t y0 = pb_hi ^ x3 ^ k0;"),
    ("philox_same_multiplier",
     "uint64_t pa = (uint64_t)PHILOX_M_A * (uint64_t)x0;",
     "uint64_t pa = (uint64_t)PHILOX_M_B * (uint64_t)x0;"),
    ("philox_low_halves_swapped", "uint32_t y1 = pb_lo;", "uint32_t y1 = pa_lo;"),
    ("counter_words_transposed",
     "{(uint32_t)b, (uint32_t)(b >> 32), region_id, 0u}",
     "{(uint32_t)b, region_id, (uint32_t)(b >> 32), 0u}"),
    # storage formats
    ("f16_subnormal_scale", "else if (ex == 0) v = ldexp((double)man, -24);",
     "else if (ex == 0) v = ldexp((double)man, -25);"),
    ("f16_exponent_bias", "ldexp((double)(1024 + man), ex - 25)",
     "ldexp((double)(1024 + man), ex - 24)"),
    ("f8_subnormal_scale", "ldexp((double)man, -9)", "ldexp((double)man, -10)"),
    ("bf16_round_half_up", "u += 0x7FFFu + lsb;", "u += 0x8000u;"),
    ("rne_ties_away", "(rem == half && (q & 1u))", "(rem == half)"),
    ("f8_overflow_to_nan", "if (bits_f32(a) >= 448.0f) return (uint8_t)(sign | 0x7Eu);",
     "if (bits_f32(a) >= 448.0f) return (uint8_t)(sign | 0x7Fu);"),
    ("f16_underflow_cut", "if (e < -25) return sign;", "if (e < -24) return sign;"),
    # Box-Muller in fp32
    ("log1p_quartic_sign", "fmaf(r, -0.25f, C_THIRD)", "fmaf(r, 0.25f, C_THIRD)"),
    ("ln2_tail_dropped", "float lo = fmaf(ef, C_LN2_LO, T_LO[j]);", "float lo = T_LO[j];"),
    ("ln_table_truncated", "int I = (32768 + den / 2) / den;", "int I = 32768 / den;"),
    ("series_sign_pattern", "if ((j / 2) % 2 == 1) c = -c;", "if (j % 2 == 1) c = -c;"),
    ("quarter_turn_truncated", "uint32_t q = (k + (1u << 21)) >> 22;", "uint32_t q = k >> 22;"),
    ("quadrant_sign", "case 1: *sn_out = cs;  *cs_out = -sn; break;",
     "case 1: *sn_out = cs;  *cs_out = sn; break;"),
    ("radius_factor_dropped", "float rho = sqrtf(-2.0f * l);", "float rho = sqrtf(-l);"),
    ("u1_offset_dropped", "oracle_ln_u24((w0 >> 8) + 1u)", "oracle_ln_u24(w0 >> 8)"),
    ("cos_sin_outputs_swapped", "*z0 = rho * cs;\n  *z1 = rho * sn;",
     "*z0 = rho * sn;\n  *z1 = rho * cs;"),
    # the 16-bit and 8-bit formats (reading R12)
    ("n16_mirror_dropped", "uint32_t t = (k & 0x7FFFu) ^ (d ? 0x7FFFu : 0u);",
     "uint32_t t = k & 0x7FFFu;"),
    ("n16_mirror_scale_dropped", "(float)(2u * t + 1u) * (d ? 65536.0f : 1.0f);",
     "(float)(2u * t + 1u) * 1.0f;"),
    ("n16_cell_bits", "(int)((b >> 19) & 15u)", "(int)((b >> 20) & 15u)"),
    ("n16_chord_width", "long double m0 = 1.0L + i / 16.0L, m1 = m0 + 1.0L / 16.0L;",
     "long double m0 = 1.0L + i / 16.0L, m1 = m0 + 1.0L / 32.0L;"),
    ("n16_u_scale", "long double y = ldexpl(m, e - 17);", "long double y = ldexpl(m, e - 16);"),
    ("angle16_half_step_dropped", "fmaf((float)n - 128.0f, C16_STEP, C16_STEP * 0.5f)",
     "fmaf((float)n - 128.0f, C16_STEP, 0.0f)"),
    ("angle16_rotation_sign", "*cs = fmaf(-T_SIN[j], delta, T_COS[j]);",
     "*cs = fmaf(T_SIN[j], delta, T_COS[j]);"),
    ("angle_table_not_midpoint", "long double phi = 2.0L * pi * (j + 0.5L) / 256.0L;",
     "long double phi = 2.0L * pi * j / 256.0L;"),
    ("n16_radius_from_high_half", "float rho = oracle_radius16(w & 0xFFFFu);",
     "float rho = oracle_radius16(w >> 16);"),
    ("n16_outputs_swapped", "*v0 = fmaf(rs, cs, mean);\n  *v1 = fmaf(rs, sn, mean);",
     "*v0 = fmaf(rs, sn, mean);\n  *v1 = fmaf(rs, cs, mean);"),
    ("n16_std_dropped", "float rs = rho * sd;\n  *v0 = fmaf(rs, cs, mean);",
     "float rs = rho;\n  *v0 = fmaf(rs, cs, mean);"),
    ("n8_bytes_swapped", "float rho = R8_RHO[h & 255u];\n  uint32_t j = (h >> 8) & 255u;",
     "float rho = R8_RHO[(h >> 8) & 255u];\n  uint32_t j = h & 255u;"),
    ("r8_quantile_not_midpoint", "logl((j + 0.5L) / 256.0L)", "logl((j + 1.0L) / 256.0L)"),
    ("n8_half_index", "(w[(i % 16) / 4] >> (16 * ((i % 4) / 2))) & 0xFFFFu",
     "(w[(i % 16) / 4] >> (16 * (i % 2))) & 0xFFFFu"),
    ("n16_word_index", "oracle_normal16(w[(i % 8) / 2], mean, sd, &v0, &v1);",
     "oracle_normal16(w[(i % 8) % 4], mean, sd, &v0, &v1);"),
    ("uniform16_scale", "& 0xFFFFu) * 0x1p-16f;", "& 0xFFFFu) * 0x1p-15f;"),
    ("uniform8_byte_order", "(w[(i % 16) / 4] >> (8 * (i % 4))) & 0xFFu",
     "(w[(i % 16) / 4] >> (8 * (3 - i % 4))) & 0xFFu"),
    # Tier-1 fill
    ("raw_big_endian", "(uint8_t)(word >> (8 * (j % 4)))", "(uint8_t)(word >> (8 * (3 - j % 4)))"),
    ("int_range_modulo", "uint64_t off = ((uint64_t)w[i % 4] * span) >> 32;",
     "uint64_t off = (uint64_t)w[i % 4] % span;"),
    ("uniform_sign", "float v = lo + f * width;", "float v = lo - f * width;"),
    ("uniform_fraction_bits", "f = (float)(w[i % 4] >> 8) * 0x1p-24f;",
     "f = (float)(w[i % 4] >> 9) * 0x1p-23f;"),
    ("normal_pair_index", "unsigned pair = (unsigned)((i % 4) / 2);",
     "unsigned pair = (unsigned)((i % 4) % 2);"),
    ("normal_affine_order", "float v = mean + sd * z;", "float v = sd + mean * z;"),
    ("guard_band_misplaced", "uint8_t *hi = alloc + glo + payload_bytes;",
     "uint8_t *hi = alloc + payload_bytes;"),
    # guard check and the equivalence predicate
    ("guard_first_relative", "first = base + j;", "first = j;"),
    ("guard_hi_base", "uint64_t base = (uint64_t)glo + payload_bytes;",
     "uint64_t base = payload_bytes;"),
    ("guards_of_reference_reported",
     "oracle_guard_check(cand_alloc, bytes, cand_glo, cand_ghi, cand_canary, &gbad, &gfirst);",
     "oracle_guard_check(ref_alloc, bytes, cand_glo, cand_ghi, cand_canary, &gbad, &gfirst);"),
    ("nan_pair_mismatch", "if (isnan(r) && isnan(c)) mismatch = 0;", "if (0) mismatch = 0;"),
    ("inf_sign_ignored", "isinf(r) && isinf(c) && (signbit(r) == signbit(c))",
     "isinf(r) && isinf(c)"),
    ("bound_on_candidate", "double bound = atol + rtol * fabs(r);",
     "double bound = atol + rtol * fabs(c);"),
    ("bound_inclusive", "mismatch = d > bound;", "mismatch = d >= bound;"),
    ("rel_on_candidate", "if (r != 0.0) rel_err = d / fabs(r);",
     "if (r != 0.0) rel_err = d / fabs(c);"),
    ("rel_zero_reference", "else rel_err = (d == 0.0) ? 0.0 : INFINITY;",
     "else rel_err = d;"),
    ("last_mismatch_kept", "if (st.first_mismatch == UINT64_MAX) st.first_mismatch = i;",
     "st.first_mismatch = i;"),
    ("int_compare_one_sided", "(size_t)sz) != 0;", "(size_t)sz) > 0;"),
    ("nonfinite_not_counted", "else { mismatch = 1; st.nonfinite_mismatches += 1; }",
     "else { mismatch = 1; }"),
    # the exact sums of the Eq. 1 cosine
    ("eq_cc_uses_cross_product", "eq_add(cc, c * c);", "eq_add(cc, r * c);"),
    ("eq_rr_uses_cross_product", "eq_add(rr, r * r);", "eq_add(rr, r * c);"),
    ("eq_rr_needs_finite_pair", "if (isfinite(r)) eq_add(rr, r * r);",
     "if (isfinite(r) && isfinite(c)) eq_add(rr, r * r);"),
    ("eq_top_digit_dropped", "acc[q + 2] += sg * (int64_t)hi;", ""),
    ("eq_sign_dropped", "int64_t sg = (p < 0.0) ? -1 : 1;", "int64_t sg = 1;"),
    ("eq_lsb_off_by_one", "int lsb = e - 53;", "int lsb = e - 52;"),
    ("eq_mid_digit_shift", "((m >> (32 - b)) & 0xFFFFFFFFu)", "((m >> (31 - b)) & 0xFFFFFFFFu)"),
    # the exact sums of binary64 regions
    ("eq64_digit_shift_off_by_one", "(int64_t)eq64_bits(M, 32 * k - b);",
     "(int64_t)eq64_bits(M, 32 * k - b - 1);"),
    ("eq64_top_digit_dropped", "for (int k = 0; k < 5; ++k) {\n    int64_t dig",
     "for (int k = 0; k < 4; ++k) {\n    int64_t dig"),
    ("eq64_low_bits_shifted_away", "if (lo < 0) return (uint64_t)((M << -lo) & 0xFFFFFFFFu);",
     "if (lo < 0) return (uint64_t)((M >> -lo) & 0xFFFFFFFFu);"),
    ("eq64_cross_sign_of_reference", "eq64_add(rc, nr != nc, mr, er, mc, ec);",
     "eq64_add(rc, nr, mr, er, mc, ec);"),
    ("eq64_rr_uses_candidate", "eq64_add(rr, 0, mr, er, mr, er);", "eq64_add(rr, 0, mr, er, mc, ec);"),
    ("eq64_cc_needs_finite_pair", "if (isfinite(c)) eq64_add(cc, 0, mc, ec, mc, ec);",
     "if (isfinite(r) && isfinite(c)) eq64_add(cc, 0, mc, ec, mc, ec);"),
    ("eq64_exponent_off_by_one", "int ee = ex - 53;", "int ee = ex - 52;"),
    # further stored formats
    ("fnuz_negative_zero_kept", "if (fnuz && mag == 0) return 0;", ""),
    ("e5m2_saturates_to_inf", "encode_fp8(f, 5, 2, 15, 0x7Bu, 0)", "encode_fp8(f, 5, 2, 15, 0x7Cu, 0)"),
    ("e4m3fnuz_encoder_bias", "encode_fp8(f, 4, 3, 8, 0x7Fu, 1)", "encode_fp8(f, 4, 3, 7, 0x7Fu, 1)"),
    ("e5m2fnuz_decoder_bias", "ldexp((double)(4 + man), ex - 18)", "ldexp((double)(4 + man), ex - 17)"),
    ("e4m3fnuz_nan_pattern", "double oracle_decode_f8e4m3fnuz(uint8_t b) {\n  if (b == 0x80u) return NAN;",
     "double oracle_decode_f8e4m3fnuz(uint8_t b) {\n  if (b == 0xFFu) return NAN;"),
    ("i64_difference_rounded_late", "abs_err = (double)(unsigned __int128)dd;",
     "abs_err = fabs((double)c - (double)r);"),
    ("restore_guards_skipped", "oracle_fill_guards(alloc, payload_bytes, glo, ghi, canary);\n  memcpy",
     "memcpy"),
]


def _params(fn):
    """Every argument binding of a test function's parametrize marks."""
    axes = []
    for m in getattr(fn, "pytestmark", []):
        if m.name != "parametrize":
            continue
        names, values = m.args[0], m.args[1]
        names = [n.strip() for n in names.split(",")] if isinstance(names, str) else list(names)
        rows = []
        for v in values:
            if hasattr(v, "values") and hasattr(v, "marks"):     # pytest.param(...)
                v = tuple(v.values)
            elif len(names) == 1:
                v = (v,)
            rows.append(dict(zip(names, v)))
        axes.append(rows)
    for combo in itertools.product(*axes):
        kw = {}
        for d in combo:
            kw.update(d)
        yield kw


def _pins(torch_philox, cheap_only=False):
    """(label, zero-argument callable) for every pin, cheapest first."""
    found = []
    for modname in PIN_MODULES:
        mod = importlib.import_module(modname)
        for name, fn in vars(mod).items():
            if not name.startswith("test_") or not callable(fn):
                continue
            if cheap_only and name in EXPENSIVE:
                continue
            argnames = fn.__code__.co_varnames[:fn.__code__.co_argcount]
            for kw in _params(fn):
                call = dict(kw)
                if "oracle" in argnames:
                    call["oracle"] = O
                if "torch_philox" in argnames:
                    call["torch_philox"] = torch_philox
                label = "%s::%s%s" % (modname.split(".")[-1], name,
                                      sorted(kw.items()) if kw else "")
                rank = EXPENSIVE.index(name) + 1 if name in EXPENSIVE else 0
                found.append((rank, len(found), label, fn, call))
    found.sort(key=lambda t: (t[0], t[1]))
    return [(label, (lambda f=fn, c=call: f(**c))) for _, _, label, fn, call in found]


def _first_failing_pin(pins):
    for label, run in pins:
        try:
            run()
        except Exception as e:                      # an assertion, or a raise
            return label, type(e).__name__
    return None


@pytest.fixture(scope="module")
def source():
    with open(oracle_build.SRC) as f:
        return f.read()


def _compile(tmp_path, text, name):
    src = tmp_path / (name + ".c")
    src.write_text(text)
    return oracle_build.compile_library(str(src), str(tmp_path / ("lib" + name + ".so")))


def test_runner_passes_the_unmodified_oracle(tmp_path, source, torch_philox):
    """The same runner on an unmodified copy: every (cheap) pin passes, so a
    failure below is the planted mistake's doing."""
    pins = _pins(torch_philox, cheap_only=True)
    assert len(pins) > 60
    with O.use_library(_compile(tmp_path, source, "pristine")):
        assert _first_failing_pin(pins) is None


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_fails_a_pin(tmp_path, source, torch_philox, name, old, new):
    assert source.count(old) == 1, "mutation site of %s not unique" % name
    path = _compile(tmp_path, source.replace(old, new), name)
    with O.use_library(path):
        caught = _first_failing_pin(_pins(torch_philox))
    assert caught is not None, "no pin fails with the mutant %s" % name
    os.remove(path)
