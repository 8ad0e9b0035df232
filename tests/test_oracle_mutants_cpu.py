"""The oracle's pins catch plausible mistakes in the oracle itself.

Each mutant below plants one mistake (a dropped term, a wrong sign, index,
operand or rounding) into a scratch copy of ``oracle/`` and runs the CPU pin
suites (closed forms, library special cases, brute force, stored fixtures)
against it; every mutant must fail at least one pin.  The unmutated copy
must pass them all (the harness itself is sound).  Nothing here touches the
CUDA path.
"""
import os
import shutil
import subprocess
import sys
import tempfile
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PIN_SUITES = ["tests/test_oracle_pins.py", "tests/test_synth_and_golden.py", "tests/test_attention_oracle.py",
              "tests/test_rope_oracle.py"]

G = "oracle/wq4_oracle.c"
AT = "oracle/attention_oracle.c"
CH = "oracle/chain.py"
PY = "oracle/__init__.py"

# (name, file, text, replacement, occurrence of the text: None = it must be unique)
MUTANTS = [
    # fp16 codec and ulp
    ("decode exponent bias", G, "exp - 25)", "exp - 24)", None),
    ("decode subnormal scale", G, "ldexp((double)man, -24)", "ldexp((double)man, -25)", None),
    ("encode ties away from zero", G, "double m = nearbyint(ldexp(f, 11));", "double m = round(ldexp(f, 11));", None),
    ("encode subnormal truncates", G, "nearbyint(ldexp(a, 24))", "floor(ldexp(a, 24))", None),
    ("encode drops the exponent carry", G, "{ m = 1024.0; ex += 1; }", "{ m = 1024.0; }", None),
    ("ulp one binade high", G, "ldexp(1.0, (e - 1) - 10)", "ldexp(1.0, e - 10)", None),
    # the format
    ("nibble order reversed", G, "(word >> (4 * (k % 8)))", "(word >> (4 * (7 - k % 8)))", None),
    ("row index halved", G, "W[(int64_t)n * (K / 8) + k / 8]", "W[(int64_t)(n / 2) * (K / 8) + k / 8]", None),
    ("pack nibble order reversed", G, "word |= code << (4 * i);", "word |= code << (4 * (7 - i));", None),
    ("unpack zero point 6", G, "w_out[(int64_t)n * K + k] = (double)(q - 7) * sc;",
     "w_out[(int64_t)n * K + k] = (double)(q - 6) * sc;", None),
    # the GEMV
    ("zero point 8", G, "double w = (double)(q - 7) * sc;", "double w = (double)(q - 8) * sc;", None),
    ("scale dropped", G, "double w = (double)(q - 7) * sc;", "double w = (double)(q - 7);", None),
    ("scale of the next group", G, "s[(int64_t)n * (K / 32) + k / 32]", "s[(int64_t)n * (K / 32) + (k / 32 + 1) % (K / 32)]", 1),
    ("activation transposed", G, "x[(int64_t)b * K + k]", "x[(int64_t)k * batch + b]", None),
    ("magnitude without abs", G, "mag += fabs(w * xv);", "mag += w * xv;", None),
    ("row factor not applied", G, "acc *= rb;", "(void)rb;", None),
    ("row factor of the first row", G, "double rb = r ? r[b] : 1.0;", "double rb = r ? r[0] : 1.0;", None),
    ("magnitude without the row factor", G, "mag *= rb;", "(void)mag;", None),
    ("last code of a row dropped", G, "            for (int k = 0; k < K; ++k) {\n                int q = wq4o_code",
     "            for (int k = 0; k < K - 1; ++k) {\n                int q = wq4o_code", None),
    ("fp16 output rounded through fp32", G, "wq4o_double_to_half(acc)", "wq4o_double_to_half((float)acc)", None),
    # chain glue
    ("RMS without eps", G, "sqrt(ss / (double)n + eps)", "sqrt(ss / (double)n)", None),
    ("RMS mean over n - 1", G, "sqrt(ss / (double)n + eps)", "sqrt(ss / (double)(n - 1) + eps)", None),
    ("SiLU sign", G, "exp(-gv)", "exp(gv)", None),
    ("SiLU without up", G, "double v = gv / (1.0 + exp(-gv)) * uv;", "double v = gv / (1.0 + exp(-gv));", None),
    ("residual subtracts", G, "wq4o_half_to_double(a[i]) + wq4o_half_to_double(b[i])",
     "wq4o_half_to_double(a[i]) - wq4o_half_to_double(b[i])", None),
    # chain composition
    ("attention stand-in from the key block", CH, "a = np.ascontiguousarray(qkv[:, :H])",
     "a = np.ascontiguousarray(qkv[:, H:2 * H])", None),
    ("QKV without its RMS factor", CH, 'gemv(*w["qkv"], u, r1)', 'gemv(*w["qkv"], u)', None),
    ("O with the layer input's factor", CH, 'gemv(*w["o"], a, r2)', 'gemv(*w["o"], a, r1)', None),
    ("residual from u instead of v", CH, "x1 = add_fp16(v, o)", "x1 = add_fp16(u, o)", None),
    ("gate_up on v instead of x1", CH, 'gemv(*w["gate_up"], x1, r3)', 'gemv(*w["gate_up"], v, r3)', None),
    ("gate and up swapped", CH, "silu_mul(np.ascontiguousarray(gu[:, :F]), np.ascontiguousarray(gu[:, F:]))",
     "silu_mul(np.ascontiguousarray(gu[:, F:]), np.ascontiguousarray(gu[:, :F]))", None),
    ("down normalised", CH, 'gemv(*w["down"], m)', 'gemv(*w["down"], m, rms_factors(m, eps))', None),
    ("second residual from v", CH, "x2 = add_fp16(x1, d)", "x2 = add_fp16(v, d)", None),
    ("LM head without its RMS factor", CH, "gemv(*lm_head, x, rf)", "gemv(*lm_head, x)", None),
    # attention
    ("query of the kv head", AT, "const uint16_t* qj = q + (int64_t)b * q_stride + (int64_t)j * head_dim;",
     "const uint16_t* qj = q + (int64_t)b * q_stride + (int64_t)h * head_dim;", None),
    ("attention output rounded through fp32", AT, "o16j[d] = wq4o_double_to_half(oj[d]);",
     "o16j[d] = wq4o_double_to_half((float)oj[d]);", None),
    ("maximum of the unscaled scores", AT, "const double st = scale * dot;", "const double st = dot;", None),
    ("kv head by modulo", AT, "const int h = j / G;", "const int h = j % n_kv_heads;", None),
    ("scale dropped in the weights", AT, "exp(scale * dot - m)", "exp(dot - m)", None),
    ("no max shift", AT, "exp(scale * dot - m)", "exp(scale * dot)", None),
    ("attention magnitude without abs", AT, "Aj[d] += e * fabs(v);", "Aj[d] += e * v;", None),
    ("normaliser off by one", AT, "oj[d] /= Z;", "oj[d] /= (Z + 1.0);", None),
    ("length one short", AT, "const int T = seq_lens[b] > 0 ? seq_lens[b] : 0;",
     "const int T = seq_lens[b] > 1 ? seq_lens[b] - 1 : 0;", 1),
    ("value row shifted", AT,
     "const uint16_t* vt = cache_row(v_cache, n_kv_heads, page_size, head_dim, page, h, t % page_size);",
     "const uint16_t* vt = cache_row(v_cache, n_kv_heads, page_size, head_dim, page, h, (t + 1) % page_size);", None),
    ("value row of the key row's page", AT,
     "const uint16_t* vt = cache_row(v_cache, n_kv_heads, page_size, head_dim, page, h, t % page_size);",
     "const uint16_t* vt = cache_row(v_cache, n_kv_heads, page_size, head_dim, 0, h, t % page_size);", None),
    ("append row shifted", AT, "pos % page_size) * head_dim", "(pos + 1) % page_size) * head_dim", None),
    ("append copies head 0 everywhere", AT, "(int64_t)h * head_dim;", "(int64_t)0 * head_dim;", None),
    # rotary embedding
    ("RoPE cross-term sign", PY, "re * c - im * s", "re * c + im * s", None),
    ("RoPE frequency exponent halved", PY, "-2.0 * i / head_dim", "-1.0 * i / head_dim", None),
    ("RoPE rotate-half pairing", PY,
     "v = half_to_double(x).reshape(batch, n // head_dim, head_dim // 2, 2)",
     "v = half_to_double(x).reshape(batch, n // head_dim, 2, head_dim // 2).swapaxes(-1, -2)", None),
    ("RoPE position of row 0 for every row", PY,
     "pos = np.asarray(positions, np.float64).reshape(batch, 1, 1)",
     "pos = np.full((batch, 1, 1), float(np.asarray(positions).reshape(-1)[0]))", None),
    ("RoPE position off by one", PY, "pos = np.asarray(positions, np.float64)",
     "pos = 1.0 + np.asarray(positions, np.float64)", None),
    # the chain's attention step
    ("queries not rotated", CH, 'q64, q = rope(np.ascontiguousarray(qkv[:, :H]), pos, D, attn["theta"])',
     'q = np.ascontiguousarray(qkv[:, :H]); q64 = None', None),
    ("keys not rotated", CH, 'k64, k = rope(np.ascontiguousarray(qkv[:, H:H + Hkv * D]), pos, D, attn["theta"])',
     'k = np.ascontiguousarray(qkv[:, H:H + Hkv * D]); k64 = None', None),
    ("values from the key block", CH, "v = np.ascontiguousarray(qkv[:, H + Hkv * D:H + 2 * Hkv * D])",
     "v = np.ascontiguousarray(qkv[:, H:H + Hkv * D])", None),
    ("sequence without the new token", CH, "pos + 1,", "pos,", None),
    ("O on the query block", CH, "a = attention_step(qkv, H, attn, t)",
     "attention_step(qkv, H, attn, t); a = np.ascontiguousarray(qkv[:, :H])", None),
]


def _tree(dst):
    """The oracle, the pin suites and the seeded generator, copied to dst."""
    os.makedirs(os.path.join(dst, "oracle"))
    for f in ("__init__.py", "chain.py", "wq4_oracle.c", "attention_oracle.c"):
        shutil.copy(os.path.join(ROOT, "oracle", f), os.path.join(dst, "oracle", f))
    os.makedirs(os.path.join(dst, "tests"))
    for f in ["conftest.py"] + [os.path.basename(s) for s in PIN_SUITES]:
        shutil.copy(os.path.join(ROOT, "tests", f), os.path.join(dst, "tests", f))
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(dst, "tests", "golden"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    os.makedirs(os.path.join(dst, "paper_2412_15803_gb300"))
    for f in ("__init__.py", "synth.py"):
        shutil.copy(os.path.join(ROOT, "paper_2412_15803_gb300", f), os.path.join(dst, "paper_2412_15803_gb300", f))


def _mutate(path, text, repl, nth):
    src = open(path).read()
    n = src.count(text)
    if nth is None:
        assert n == 1, f"{text!r} occurs {n} times"
        src = src.replace(text, repl)
    else:
        assert n > nth, f"{text!r} occurs {n} times"
        at = -1
        for _ in range(nth + 1):
            at = src.index(text, at + 1)
        src = src[:at] + repl + src[at + len(text):]
    open(path, "w").write(src)


def _run_pins(mutant):
    """Exit status of the pin suites on a copy carrying `mutant` (None: unmutated)."""
    with tempfile.TemporaryDirectory(prefix="wq4_mutant_") as d:
        _tree(d)
        if mutant is not None:
            _, f, text, repl, nth = mutant
            _mutate(os.path.join(d, f), text, repl, nth)
        env = dict(os.environ, PYTHONDONTWRITEBYTECODE="1")
        cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-m", "not gpu", "-p", "no:cacheprovider", *PIN_SUITES]
        try:
            r = subprocess.run(cmd, cwd=d, env=env, capture_output=True, text=True, timeout=600)
        except subprocess.TimeoutExpired:
            return -1, "timeout"
        return r.returncode, r.stdout[-2000:] + r.stderr[-2000:]


def test_mutant_texts_apply():
    """Every planted mistake names text that exists in the current oracle."""
    for name, f, text, _, nth in MUTANTS:
        n = open(os.path.join(ROOT, f)).read().count(text)
        assert (n == 1) if nth is None else (n > nth), (name, n)


def test_every_mutant_fails_a_pin():
    workers = max(1, min(8, os.cpu_count() or 1))
    with ThreadPoolExecutor(max_workers=workers) as ex:
        control = ex.submit(_run_pins, None)
        results = list(ex.map(_run_pins, MUTANTS))
    rc, out = control.result()
    assert rc == 0, "the unmutated copy fails its pins:\n" + out
    survivors = [m[0] for m, (rc, _) in zip(MUTANTS, results) if rc == 0]
    assert not survivors, f"mutants no pin catches: {survivors}"
