"""Plant plausible mistakes in copies of the oracle and check that the pins
catch every one of them (a dropped term, a wrong sign, index or offset, a
transposed operand, a broken tie rule ...).  The mistakes are planted in the C
source of the CPU oracle only, built into separate libraries under a temporary
directory, and checked in a subprocess."""
import json
import os
import subprocess
import sys

import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))

# (name, [(exact text in cci_oracle.c, replacement), ...])
MUTANTS = [
    ("tie_to_higher_index", [("order[pos - 1]) * R + r]) < a)", "order[pos - 1]) * R + r]) <= a)")]),
    ("keeps_smallest", [("order[pos - 1]) * R + r]) < a)", "order[pos - 1]) * R + r]) > a)")]),
    ("signed_not_magnitude", [("double a = fabs(W[(gi * G + j) * R + r]);", "double a = W[(gi * G + j) * R + r];"),
                              ("fabs(W[(gi * G + order[pos - 1]) * R + r])", "W[(gi * G + order[pos - 1]) * R + r]")]),
    ("emit_descending", [("kept[p - 1] > v", "kept[p - 1] < v")]),
    ("idx_from_rank_order", [("idx[o] = (uint8_t)kept[s];", "idx[o] = (uint8_t)order[s];")]),
    ("nan_accepted", [("if (isnan(W[e])) return OR_VALUE;", ";")]),
    ("group_offset_K", [("const int64_t co = gi * G + idx[o];", "const int64_t co = gi * K + idx[o];")]),
    ("duplicates_overwrite", [("Wd[co * R + r] += values[o];", "Wd[co * R + r] = values[o];")]),
    ("linear_drops_last_term", [("for (int64_t r = 0; r < R; ++r) {\n                if (!mask",
                                 "for (int64_t r = 0; r < R - 1; ++r) {\n                if (!mask")]),
    ("linear_sign", [("acc += Wd[co * R + r] * X[n * R + r];", "acc -= Wd[co * R + r] * X[n * R + r];")]),
    ("scale_signed", [("sc += fabs(Wd[co * R + r]) * fabs(X[n * R + r]);", "sc += Wd[co * R + r] * X[n * R + r];")]),
    ("alg2_group_offset", [("const int64_t row = G * i + idx[o];", "const int64_t row = K * i + idx[o];")]),
    ("conv_pad_sign", [("const int64_t h = p * sh - ph + kh;", "const int64_t h = p * sh + ph + kh;")]),
    ("conv_stride_mixup", [("const int64_t w = q * sw - pw + kw;", "const int64_t w = q * sh - pw + kw;")]),
    ("conv_tap_order", [("const int64_t r = ((int64_t)kh * KW + kw) * Cin + ci;",
                         "const int64_t r = ((int64_t)kw * KH + kh) * Cin + ci;")]),
    ("conv_out_size", [("const int64_t P = (H + 2 * ph - KH) / sh + 1;", "const int64_t P = (H + ph - KH) / sh + 1;")]),
    ("conv_skips_taps", [("if (w < 0 || w >= Wi) continue;", "if (w <= 0 || w >= Wi) continue;")]),
]


def test_mutants_are_caught(tmp_path):
    with open(oracle.SOURCE) as f:
        src = f.read()
    libs = {}
    for name, edits in MUTANTS:
        text = src
        for old, new in edits:
            assert text.count(old) == 1, (name, old)
            text = text.replace(old, new)
        path = tmp_path / f"{name}.c"
        path.write_text(text)
        libs[name] = oracle.build(force=True, src=str(path), out=str(tmp_path / f"lib{name}.so"))
    libs["unmodified"] = oracle.build(force=True, src=oracle.SOURCE,
                                      out=str(tmp_path / "libunmodified.so"))
    proc = subprocess.run([sys.executable, os.path.join(HERE, "oracle_pins.py"), *libs.values()],
                          capture_output=True, text=True, timeout=600)
    assert proc.returncode == 0, proc.stderr[-2000:]
    report = json.loads(proc.stdout.strip().splitlines()[-1])
    assert report[libs["unmodified"]] == []
    missed = [name for name, lib in libs.items() if name != "unmodified" and not report[lib]]
    assert not missed, f"mutants not caught by any pin: {missed}"
