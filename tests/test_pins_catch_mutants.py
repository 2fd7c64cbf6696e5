"""The oracle's pins catch plausible mistakes in the oracle.

Each mutant below is a copy of oracle/wq_oracle.c with one planted mistake
(a dropped term, a wrong sign, a transposed operand or index, a wrong bit
position, a wrong rounding).  The copy is compiled with the oracle's own
flags, the oracle pin tests (tests/test_oracle_*.py) run against it in a
subprocess, and they must fail.  An unmutated copy compiled the same way must
pass.  Every mutated index stays inside its array, so a mutant fails the
pins and never crashes.  All of this runs on the CPU.
"""
import glob
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor


ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "wq_oracle.c")
WORK = os.path.join(ROOT, "oracle", "_build", "mutants")

# (name, text in the source, its replacement, which occurrence: an index or "all")
MUTANTS = [
    ("zero point not rounded",
     "float zf = fminf(fmaxf(rintf(negmn_over_s), 0.0f), qmax) + 0.0f;",
     "float zf = fminf(fmaxf(negmn_over_s, 0.0f), qmax) + 0.0f;", 0),
    ("zero point subtracted from the codes",
     "float qf = fminf(fmaxf(rintf(ratio) + zf, 0.0f), qmax);",
     "float qf = fminf(fmaxf(rintf(ratio) - zf, 0.0f), qmax);", 0),
    ("group minimum taken as a maximum", "mn = fminf(mn, wg[i]);", "mn = fmaxf(mn, wg[i]);", 0),
    ("constant group keeps a zero scale", "if (orc_f16_to_f64(s16) == 0.0) s16 = 0x3C00u; /* 1.0 */", "", 0),
    ("qmax off by one", "const float qmax = (float)((1 << bits) - 1);", "const float qmax = (float)(1 << bits);", 0),
    ("scale divides by 2^bits", "volatile float s32 = range / qmax;", "volatile float s32 = range / (qmax + 1.0f);", 0),
    ("fp16 conversion truncates",
     "double r = rint(a / quantum) * quantum;   /* exact scaling, ties-even */",
     "double r = floor(a / quantum) * quantum;", 0),
    ("bf16 conversion truncates",
     "double r = rint(a / quantum) * quantum;\n    if (r >= ldexp(1.0, 128))",
     "double r = trunc(a / quantum) * quantum;\n    if (r >= ldexp(1.0, 128))", 0),
    ("fp16 subnormals off by two", "if (ex == 0) v = ldexp((double)mant, -24);",
     "if (ex == 0) v = ldexp((double)mant, -25);", 0),
    ("bf16 decode shifted", "uint32_t bits = (uint32_t)b << 16;", "uint32_t bits = (uint32_t)b << 15;", 0),
    ("2-bit bit classes swapped (pack and unpack)",
     "bit = 16 * half + 8 * (i / 8) + 2 * (2 * ((c % 32) / 16) + (c % 16) / 8);",
     "bit = 16 * half + 8 * (i / 8) + 2 * (((c % 32) / 16) + 2 * ((c % 16) / 8));", "all"),
    ("4-bit k-steps reversed (pack and unpack)",
     "word = (c / 64) * 128 + lane * 4 + (c % 64) / 16;",
     "word = (c / 64) * 128 + lane * 4 + 3 - (c % 64) / 16;", "all"),
    ("lane from the wrong feature bits (pack and unpack)",
     "const int lane = (i % 8) * 4 + (c % 8) / 2;", "const int lane = (i % 8) * 4 + (c % 4);", "all"),
    ("3-bit upper plane ignores the row half (pack and unpack)",
     "8 * ((c / 32) % 2) + 2 * cls + i / 8)", "8 * ((c / 32) % 2) + 2 * cls)", "all"),
    ("zero stored in the scale slot",
     "meta[base + 4 * e + 2 + hi] = z[(size_t)r * ngk + j];",
     "meta[base + 4 * e + 0 + hi] = z[(size_t)r * ngk + j];", 0),
    ("dequantization adds the zero point",
     "orc_f16_to_f64(s[gi]) * ((double)q[(size_t)r * k + col] - orc_f16_to_f64(z[gi]))",
     "orc_f16_to_f64(s[gi]) * ((double)q[(size_t)r * k + col] + orc_f16_to_f64(z[gi]))", 0),
    ("dot products drop the zero point",
     "const double w = orc_f16_to_f64(srow[j]) * ((double)qrow[col] - orc_f16_to_f64(zrow[j]));",
     "const double w = orc_f16_to_f64(srow[j]) * ((double)qrow[col]);", "all"),
    ("RMSNorm over the sum of squares", "rs[t] = 1.0 / sqrt(ss / d + eps);", "rs[t] = 1.0 / sqrt(ss + eps);", 0),
    ("RMSNorm without eps", "rs[t] = 1.0 / sqrt(ss / d + eps);", "rs[t] = 1.0 / sqrt(ss / d);", 0),
    ("LoRA A applied to the unnormalized input",
     "acc += xin[(size_t)tk * d + c] * orc_bf16_to_f64(lora_a[(size_t)p * d + c]);",
     "acc += orc_bf16_to_f64(x[(size_t)tk * d + c]) * orc_bf16_to_f64(lora_a[(size_t)p * d + c]);", 0),
    ("prenorm ignored", "if (prenorm) orc_rms_scale(x, m, d, eps, rs);", "if (prenorm) {}", 0),
    ("LoRA A transposed",
     "acc += xin[(size_t)tk * d + c] * orc_bf16_to_f64(lora_a[(size_t)p * d + c]);",
     "acc += xin[(size_t)tk * d + c] * orc_bf16_to_f64(lora_a[(size_t)c * 2 * r + p]);", 0),
    ("LoRA B of gate transposed",
     "lg += t[(size_t)tk * 2 * r + p] * orc_bf16_to_f64(lora_bg[(size_t)n * r + p]);",
     "lg += t[(size_t)tk * 2 * r + p] * orc_bf16_to_f64(lora_bg[(size_t)p * inter + n]);", 0),
    ("up adapter reads the gate's rows of A",
     "lu += t[(size_t)tk * 2 * r + r + p] * orc_bf16_to_f64(lora_bu[(size_t)n * r + p]);",
     "lu += t[(size_t)tk * 2 * r + p] * orc_bf16_to_f64(lora_bu[(size_t)n * r + p]);", 0),
    ("LoRA scale dropped", "g += lora_scale * lg;", "g += lg;", 0),
    ("SiLU sign", "const double h = g / (1.0 + exp(-g)) * u;", "const double h = g / (1.0 + exp(g)) * u;", 0),
    ("4-bit down subtracts the residual",
     "if (residual) y += orc_bf16_to_f64(residual[(size_t)tk * d + c]);",
     "if (residual) y -= orc_bf16_to_f64(residual[(size_t)tk * d + c]);", 0),
    ("bf16 down subtracts the residual",
     "if (residual) y += orc_bf16_to_f64(residual[(size_t)tk * d + c]);",
     "if (residual) y -= orc_bf16_to_f64(residual[(size_t)tk * d + c]);", 1),
    ("bf16 down weights transposed", "orc_bf16_to_f64(wd[(size_t)c * inter + n]);",
     "orc_bf16_to_f64(wd[(size_t)n * d + c]);", 0),
    ("attention scores not scaled by sqrt(hd)", "s[j] = dot / sqrt((double)hd);", "s[j] = dot / (double)hd;", 0),
    ("query heads interleaved over the key/value heads", "const int g = h / rep;", "const int g = h % n_kv;", 0),
    ("softmax not normalized", "oh[e] = acc / den;", "oh[e] = acc;", 0),
    ("RoPE rotates the wrong way", "v[i] = x0 * c - x1 * s;", "v[i] = x0 * c + x1 * s;", 0),
    ("RoPE frequency exponent halved", "pow(theta, -2.0 * i / hd)", "pow(theta, -1.0 * i / hd)", 0),
    ("merge drops alpha", "w_out[(size_t)row * k + col] = (float)(w + lora_scale * ba);",
     "w_out[(size_t)row * k + col] = (float)(w + ba);", 0),
    ("merge A transposed", "orc_bf16_to_f64(lora_a[(size_t)rho * k + col]);",
     "orc_bf16_to_f64(lora_a[(size_t)col * r + rho]);", 0),
]


def _mutate(text, old, new, which):
    n = text.count(old)
    assert n >= 1, f"mutation site not found: {old!r}"
    if which == "all":
        return text.replace(old, new)
    assert which < n, (old, which, n)
    at = -1
    for _ in range(which + 1):
        at = text.index(old, at + 1)
    return text[:at] + new + text[at + len(old):]


def _run_pins(lib_path):
    """Exit status of the oracle pin tests against the library at lib_path."""
    pins = sorted(glob.glob(os.path.join(ROOT, "tests", "test_oracle_*.py")))
    env = dict(os.environ, WQ_ORACLE_LIB=lib_path, OMP_NUM_THREADS="1")
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", "-m", "not gpu", *pins]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode, (r.stdout + r.stderr)[-1500:]


def _build_variant(name, text):
    import oracle
    os.makedirs(WORK, exist_ok=True)
    stem = os.path.join(WORK, name)
    with open(stem + ".c", "w") as f:
        f.write(text)
    return oracle.compile_source(stem + ".c", stem + ".so")


def test_pins_catch_every_mutant():
    text = open(SRC).read()
    jobs = [("control", text)]
    for i, (name, old, new, which) in enumerate(MUTANTS):
        jobs.append((f"m{i:02d}", _mutate(text, old, new, which)))
    libs = [(tag, _build_variant(tag, t)) for tag, t in jobs]
    with ThreadPoolExecutor(max_workers=max(1, min(8, os.cpu_count() or 1))) as ex:
        results = list(ex.map(lambda tl: _run_pins(tl[1]), libs))
    rc0, out0 = results[0]
    assert rc0 == 0, f"the unmutated copy fails its pins:\n{out0}"
    survivors = []
    for (name, *_), (rc, out) in zip(MUTANTS, results[1:]):
        if rc != 1:  # 1: some test failed; anything else is a survivor or a broken run
            survivors.append(f"{name}: pytest exit {rc}\n{out}")
    assert not survivors, "mutants the pins do not catch:\n" + "\n".join(survivors)
