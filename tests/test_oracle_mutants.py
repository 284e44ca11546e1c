"""Each plausible mistake planted in a copy of the oracle fails at least one pin.

The mutants are text edits of oracle/sn_oracle.c compiled into a temporary
library (CPU only); the oracle source itself is never modified.
"""
import os
import shutil
import subprocess

import pytest

from pins import PINS

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "sn_oracle.c")

# (name, exact text in sn_oracle.c, replacement, which occurrence (0-based))
MUTANTS = [
    ("pe_sign", "r[i] = x - te - pe;", "r[i] = x - te + pe;", 0),
    ("pe_dropped", "r[i] = x - te - pe;", "r[i] = x - te;", 0),
    ("te_dropped", "r[i] = x - te - pe;", "r[i] = x - pe;", 0),
    ("u_transposed_fwd", "c[j] += r[i] * load(U, u_dtype, (int64_t)i * k + j);",
     "c[j] += r[i] * load(U, u_dtype, (int64_t)j * d + i);", 0),
    ("u_col_reversed_bwd", "c[j] += g * load(U, u_dtype, (int64_t)i * k + j);",
     "c[j] += g * load(U, u_dtype, (int64_t)i * k + (k - 1 - j));", 0),
    ("recon_drops_te", "double x = s + pe + te;", "double x = s + pe;", 0),
    ("recon_subtracts_pe", "double x = s + pe + te;", "double x = s - pe + te;", 0),
    ("recon_wrong_c_row", "s += load(C, dtype, t * k + j) * load(U, u_dtype, (int64_t)i * k + j);",
     "s += load(C, dtype, (t + 1) % T * k + j) * load(U, u_dtype, (int64_t)i * k + j);", 0),
    ("bwd_recon_wrong_u", "s += load(C, dtype, t * k + j) * load(U, u_dtype, (int64_t)i * k + j);",
     "s += load(C, dtype, t * k + j) * load(U, u_dtype, (int64_t)((i + 1) % d) * k + j);", 1),
    ("position_div", "return pos ? (int64_t)pos[t] : t % seq_len;",
     "return pos ? (int64_t)pos[t] : t / seq_len % seq_len;", 0),
    ("position_ignores_explicit", "return pos ? (int64_t)pos[t] : t % seq_len;",
     "return t % seq_len;", 0),
    ("id_off_by_one", "int64_t id = ids[t];", "int64_t id = ids[t] + 1;", 0),
    ("vocab_check_missing", "if (id < 0 || id >= vocab)", "if (id < 0)", 0),
    ("project_skips_second_u", "s += load(U, u_dtype, i * k + j) * A[(int64_t)j * cols + c];",
     "s += A[(int64_t)j * cols + c];", 0),
    ("project_transposed_w", "s += load(U, u_dtype, i * k + j) * load(W, dtype, i * ld + c);",
     "s += load(U, u_dtype, i * k + j) * load(W, dtype, c * ld + i % cols);", 0),
    ("round_truncates", "double q = nearbyint(a / ulp);", "double q = floor(a / ulp);", 0),
    ("round_via_fp32", "double q = nearbyint(a / ulp);",
     "double q = nearbyint((double)(float)a / ulp);", 0),
]


def _mutate(text, old, new, occurrence):
    start = -1
    for _ in range(occurrence + 1):
        start = text.find(old, start + 1)
        assert start >= 0, "mutation anchor not found: %r" % old
    return text[:start] + new + text[start + len(old):]


@pytest.fixture(scope="module")
def mutant_dir(tmp_path_factory):
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    return tmp_path_factory.mktemp("mutants")


@pytest.mark.parametrize("name,old,new,occ", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(name, old, new, occ, mutant_dir):
    import oracle as oracle_pkg
    from oracle import build as obuild

    text = open(SRC).read()
    src = os.path.join(mutant_dir, "sn_oracle_%s.c" % name)
    with open(src, "w") as f:
        f.write(_mutate(text, old, new, occ))
    shutil.copy(os.path.join(ROOT, "oracle", "sn_oracle.h"), os.path.join(mutant_dir, "sn_oracle.h"))
    lib = os.path.join(mutant_dir, "libsn_oracle_%s.so" % name)
    subprocess.run(["gcc", *obuild.CFLAGS, "-I", str(mutant_dir), src, "-o", lib, "-lm"],
                   check=True)
    orc = oracle_pkg.Oracle(lib)
    caught = []
    for pin in PINS:
        try:
            pin(orc)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, "mutant %s passes every pin" % name
