"""CPU: the oracle's pins catch plausible mistakes in the oracle.  Each case
plants one mistake in a copy of oracle/focus_oracle.c (a swapped operand, a
dropped term, a wrong sign, an off-by-one exponent, a wrong tie rule, a
wrong nibble order, a wrong constant, a strict mask boundary, a factor of
the wrong coefficient), builds it with the oracle's own flags, points the
oracle module at that build, and runs a fast subset of the pins of
test_oracle_pins.py: at least one of them must fail.  The same subset
passes on the unmodified source built the same way.  The oracle's Python
functions (the AdamW step, the MMA scale-tile layout, the GEMM on an
export) get the same treatment on copies of their source, each against
its own pins."""
import inspect
import os
import subprocess

import pytest

import oracle as O
import test_oracle_pins as P

SRC = os.path.join(os.path.dirname(O.__file__), "focus_oracle.c")

# (name, text in focus_oracle.c, replacement, occurrences)
MUTANTS = [
    ("dequantized by the relaxed scale", "yv = focus_oracle_e2m1_value(code) * s_dq;",
     "yv = focus_oracle_e2m1_value(code) * s_q;", 1),
    ("dL/dc_i without the c_i^k factor", "ksum_add(&gc, G * (double)d);", "ksum_add(&gc, G);", 1),
    ("coefficient gradient sign", "double G = -ksum_value(&T) / (ce * ce);",
     "double G = ksum_value(&T) / (ce * ce);", 1),
    ("coefficient gradient over c_eff, not c_eff^2", "double G = -ksum_value(&T) / (ce * ce);",
     "double G = -ksum_value(&T) / ce;", 1),
    ("E8M0 ceiling off by one at powers of two", "e = (f == 0.5) ? E - 1 : E;", "e = E;", 1),
    ("E2M1 ties away from the even code", "(d == bestd && (c & 1) == 0)", "(d == bestd)", 2),
    ("even element in the high nibble", "if ((col & 1) == 0) *p = (uint8_t)((*p & 0xF0) | code);",
     "if ((col & 1) == 1) *p = (uint8_t)((*p & 0xF0) | code);", 1),
    ("alpha constant", "*alpha_out = amax / 2688.0f;", "*alpha_out = amax / 2687.0f;", 1),
    ("relaxed scale divided by the coefficients (Eq. 6 inverted)", "float s_q = s_dq * c_eff;",
     "float s_q = s_dq / c_eff;", 2),
    ("E4M3 exponent bias", "ldexp(1.0 + m / 8.0, e - 7)", "ldexp(1.0 + m / 8.0, e - 8)", 1),
    ("STE ratio inverted", "float rho = dead ? 0.0f : s_dq / s_q;", "float rho = dead ? 0.0f : s_q / s_dq;", 1),
    ("clipped STE mask strict at |u| = 6", "if (ste == OR_STE_CLIPPED) mask = fabsf(u) <= 6.0f;",
     "if (ste == OR_STE_CLIPPED) mask = fabsf(u) < 6.0f;", 1),
    ("clipped STE mask never applied", "if (ste == OR_STE_CLIPPED) mask = fabsf(u) <= 6.0f;",
     "if (ste == -1) mask = fabsf(u) <= 6.0f;", 1),
    ("shared-row CRS gradient times c instead of c^k", "ksum_add(&acc_c[j], G * (double)d);",
     "ksum_add(&acc_c[j], G * (double)c);", 1),
    ("shared-row DGS gradient without c", "ksum_add(&acc_d[j * K + k], G * (double)c);",
     "ksum_add(&acc_d[j * K + k], G);", 1),
    ("S^fp gradient: sign of the x / S^q term", "ksum_add(&gs, gq - gu);", "ksum_add(&gs, gq + gu);", 1),
    ("S^fp gradient: the STE term ignores the mask", "double gu = mask ? (double)gv * (double)xv / sq_exact : 0.0;",
     "double gu = (double)gv * (double)xv / sq_exact;", 1),
    ("S^fp gradient without alpha (NVFP4)", "double ds = (fmt == OR_NVFP4) ? (double)alpha : 1.0;",
     "double ds = 1.0;", 1),
    ("OCP floor rule off by one", "e = (E - 1) - 2;", "e = E - 2;", 1),
    ("NVFP4 scale denominator without the 6", "float den = alpha * 6.0f;", "float den = alpha * 4.0f;", 1),
    ("bf16 rounding ties away from even", "return (uint16_t)((b + 0x7FFFu + lsb) >> 16);",
     "return (uint16_t)((b + 0x8000u) >> 16);", 1),
    ("binary16 rounding ties up", "return fmod(f, 2.0) != 0.0 ? f + 1.0 : f;", "return f + 1.0;", 1),
    ("binary16 subnormals one binade off", "if (e == 0) v = ldexpf((float)m, -24);",
     "if (e == 0) v = ldexpf((float)m, -25);", 1),
    ("dequantization with swapped nibbles", "int code = (col & 1) ? (byte >> 4) : (byte & 15);",
     "int code = (col & 1) ? (byte & 15) : (byte >> 4);", 1),
    ("NVFP4 dequantization without alpha", ": focus_oracle_e4m3_decode(sb) * alpha;",
     ": focus_oracle_e4m3_decode(sb);", 1),
]

# fast pins (a few seconds together), with their parameters
PINS = [
    (P.test_hand_mxfp4_block_crs, ()),
    (P.test_hand_gx_rounding_order, ()),
    (P.test_hand_mxfp4_ties, ()),
    (P.test_hand_nvfp4_blocks, ()),
    (P.test_alpha_closed_form, ()),
    (P.test_e4m3_decode_matches_torch, ()),
    (P.test_e2m1_brute_force_grid, ()),
    (P.test_e8m0_ceil_and_floor_rules, ()),
    (P.test_crs_at_one_equals_rtn, (O.MXFP4,)),
    (P.test_crs_at_one_equals_rtn, (O.NVFP4,)),
    (P.test_dequant_of_export_equals_forward, (O.MXFP4, "f32")),
    (P.test_dequant_of_export_equals_forward, (O.NVFP4, "bf16")),
    (P.test_input_gradient_is_g_over_c, (O.MXFP4,)),
    (P.test_coefficient_gradients_finite_difference, (O.NVFP4, 8)),
    (P.test_autograd_restatement, (O.MXFP4,)),
    (P.test_clipped_ste_masks_saturated, ()),
    (P.test_clipped_ste_keeps_the_saturation_boundary, ()),
    (P.test_shared_row_gradients_sum_over_rows, ()),
    (P.test_hand_mxfp4_sfp_gradient, ()),
    (P.test_hand_mxfp4_sfp_gradient_clipped_ste, ()),
    (P.test_sfp_gradient_autograd, (O.NVFP4,)),
    (P.test_bf16_rne_matches_torch, ()),
    (P.test_f16_decode_all_patterns_matches_numpy, ()),
    (P.test_f16_rne_matches_numpy, ()),
]

# planted mistakes in the oracle's Python functions:
# (name, function, text in its source, replacement)
PY_MUTANTS = [
    ("AdamW: weight decay skipped", "adamw", "p = np.asarray(p, np.float64) * (1.0 - lr * weight_decay)",
     "p = np.asarray(p, np.float64)"),
    ("AdamW: second moment without bias correction", "adamw", "vhat = v / (1.0 - beta2 ** t)", "vhat = v"),
    ("AdamW: epsilon inside the square root", "adamw", "(np.sqrt(vhat) + eps)", "np.sqrt(vhat + eps)"),
    ("AdamW: first moment with the second moment's beta", "adamw",
     "m = beta1 * np.asarray(m, np.float64) + (1.0 - beta1) * g",
     "m = beta2 * np.asarray(m, np.float64) + (1.0 - beta2) * g"),
    ("MMA scale tiles: row and column offsets swapped in a line", "mma_scale_tiles",
     "(rr % 32) * 16 + (rr // 32) * 4 + cc", "(rr % 32) * 16 + (rr // 32) + cc * 4"),
    ("GEMM: NVFP4 without the per-tensor scales", "fp4_gemm",
     "d = d * (float(np.float32(alpha_a)) * float(np.float32(alpha_b)))", "d = d"),
    ("GEMM: even element from the high nibble", "fp4_gemm", "nib[:, 0::2] = codes & 15", "nib[:, 0::2] = codes >> 4"),
    ("GEMM: E8M0 bias off by one", "fp4_gemm", "s = np.ldexp(1.0, sb.astype(np.int64) - 127)",
     "s = np.ldexp(1.0, sb.astype(np.int64) - 126)"),
]

# the pins each Python function is held to
PY_PINS = {
    "adamw": [(P.test_adamw_matches_torch, ()), (P.test_adamw_first_step_closed_form, ()),
              (P.test_bwd_adamw_equals_autograd_and_torch_adamw, (O.MXFP4,))],
    "mma_scale_tiles": [(P.test_mma_scale_tiles_hand_offsets, ()), (P.test_mma_scale_tiles_is_a_permutation, ())],
    "fp4_gemm": [(P.test_fp4_gemm_matches_independent_dequant, (O.MXFP4,)),
                 (P.test_fp4_gemm_matches_independent_dequant, (O.NVFP4,)),
                 (P.test_fp4_gemm_is_the_product_of_fake_quantized_operands, (O.NVFP4,))],
}


def build_variant(tmp, name, text):
    src = os.path.join(tmp, f"{name}.c")
    lib = os.path.join(tmp, f"lib{name}.so")
    with open(src, "w") as f:
        f.write(text)
    subprocess.check_call(["gcc", *O.CFLAGS, src, "-o", lib, "-lm"])
    return lib


def run_pins(pins):
    failed = []
    for fn, args in pins:
        try:
            fn(*args)
        except Exception as e:   # a failed assertion, or a mutant's exception
            failed.append(f"{fn.__name__}{args}: {type(e).__name__}")
    return failed


def failing_pins(lib):
    """Names of the pins in PINS that fail with the oracle loaded from lib."""
    saved = (O._LIB, O._lib)
    O._LIB, O._lib = lib, None
    try:
        return run_pins(PINS)
    finally:
        O._LIB, O._lib = saved


def py_variant(name, text, repl):
    """Oracle function `name` rebuilt from its source with one replacement,
    in the oracle module's namespace."""
    src = inspect.getsource(getattr(O, name))
    assert src.count(text) == 1, text
    ns = dict(vars(O))
    exec(src.replace(text, repl), ns)
    return ns[name]


def failing_py_pins(name, fn):
    saved = getattr(O, name)
    setattr(O, name, fn)
    try:
        return run_pins(PY_PINS[name])
    finally:
        setattr(O, name, saved)


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


def test_unmodified_source_passes_the_pins(tmp_path, source):
    assert failing_pins(build_variant(str(tmp_path), "control", source)) == []


@pytest.mark.parametrize("name,text,repl,count", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(tmp_path, source, name, text, repl, count):
    assert source.count(text) == count, (name, source.count(text))
    lib = build_variant(str(tmp_path), "mutant", source.replace(text, repl))
    failed = failing_pins(lib)
    assert failed, f"no pin caught: {name}"


@pytest.mark.parametrize("name", sorted(PY_PINS))
def test_unmodified_python_functions_pass_their_pins(name):
    assert failing_py_pins(name, py_variant(name, f"def {name}(", f"def {name}(")) == []


@pytest.mark.parametrize("name,fn,text,repl", PY_MUTANTS, ids=[m[0] for m in PY_MUTANTS])
def test_planted_python_mistake_fails_a_pin(name, fn, text, repl):
    assert failing_py_pins(fn, py_variant(fn, text, repl)), f"no pin caught: {name}"
