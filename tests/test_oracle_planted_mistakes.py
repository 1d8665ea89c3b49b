"""Planted mistakes: each alters one line of a copy of the oracle's sources, the kind of
mistake a restatement of the paper could make (a dropped term, a wrong sign, a wrong index,
a transposed operand), builds that copy into a separate library, and runs the pins of that
part of the oracle against it.  Every planted mistake must make at least one pin fail; the
unaltered copy must pass them all.  Runs on the CPU; the oracle's own sources stay as they
are.
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor
from pathlib import Path

ROOT = Path(__file__).resolve().parents[1]
sys.path.insert(0, str(ROOT))
from oracle._build import SOURCES, compile_library  # noqa: E402

PINS = {
    "gem": "tests/test_oracle_gem_pins.py",
    "mlp": "tests/test_oracle_mlp_pins.py",
    "cnn": "tests/test_oracle_cnn_pins.py",
    "schedule": "tests/test_oracle_schedule_pins.py",
    "pi": "tests/test_oracle_pi_pins.py",
}

# (name, source file, exact text, replacement, pins)
MISTAKES = [
    # the commit (Algorithm 1, Psi_GEM and Commit)
    ("moment adds -dtheta", "gem_oracle.cpp",
     "local first moment).\n    m = mu * m + dtheta;", "local first moment).\n    m = mu * m - dtheta;", "gem"),
    ("momentum term dropped", "gem_oracle.cpp",
     "local first moment).\n    m = mu * m + dtheta;", "local first moment).\n    m = dtheta;", "gem"),
    ("drift |theta + s|", "gem_oracle.cpp",
     "std::fabs(theta_pulled - s)", "std::fabs(theta_pulled + s)", "gem"),
    ("eps inside the absolute value", "gem_oracle.cpp",
     "(std::fabs(dtheta) + eps)", "std::fabs(dtheta + eps)", "gem"),
    ("no clamp of pi", "gem_oracle.cpp",
     "if (!(pi > T(0))) pi = T(0);", "", "gem"),
    ("update applied with the wrong sign", "gem_oracle.cpp",
     "theta = theta_pulled + pi * dtheta;", "theta = theta_pulled - pi * dtheta;", "gem"),
    ("pull before the commit", "gem_oracle.cpp",
     "  s = precommit_snapshot ? theta_pulled : theta;\n  return pi;",
     "  s = theta_pulled;\n  return pi;", "gem"),
    ("another worker's snapshot", "gem_oracle.cpp",
     "T* sw = s + int64_t(w) * state_stride;", "T* sw = s + int64_t((w + 1) % n) * state_stride;", "gem"),
    ("factor recorded one coordinate off", "gem_oracle.cpp",
     "if (pi_row) pi_row[j] = pi;", "if (pi_row) pi_row[j > 0 ? j - 1 : 0] = pi;", "pi"),
    # the MLP gradient
    ("bias dropped from the forward pass", "mlp_oracle.cpp",
     "z[l][int64_t(i) * ly.out + o] = acc + bias[o];", "z[l][int64_t(i) * ly.out + o] = acc;", "mlp"),
    ("ReLU derivative dropped", "mlp_oracle.cpp",
     "z[l - 1][int64_t(i) * ly.in + k] > 0.0 ? acc : 0.0;", "acc;", "mlp"),
    ("transposed weights in the backward pass", "mlp_oracle.cpp",
     "operand(W[int64_t(o) * ly.in + k], tf32);\n        prev[",
     "operand(W[int64_t(k) * ly.out + o], tf32);\n        prev[", "mlp"),
    ("softmax gradient without 1/b", "mlp_oracle.cpp",
     "delta[int64_t(i) * C + c] = (p - (c == y[i] ? 1.0 : 0.0)) / double(b);",
     "delta[int64_t(i) * C + c] = (p - (c == y[i] ? 1.0 : 0.0));", "mlp"),
    ("TF32 rounding truncates", "mlp_oracle.cpp",
     "  u += 0x00001000u;\n  u &= 0xFFFFE000u;", "  u &= 0xFFFFE000u;", "mlp"),
    ("TF32 keeps one mantissa bit too many", "mlp_oracle.cpp",
     "  u += 0x00001000u;\n  u &= 0xFFFFE000u;", "  u += 0x00000800u;\n  u &= 0xFFFFF000u;", "mlp"),
    # the CNN gradient
    ("dropout scale missing from the backward pass", "cnn_oracle.cpp",
     "da2[(size_t(co) * P2 + py) * P2 + px] * drop[int64_t(r) * n.c2 + co];",
     "da2[(size_t(co) * P2 + py) * P2 + px];", "cnn"),
    ("conv1 as a convolution (flipped kernel) instead of a correlation", "cnn_oracle.cpp",
     "acc += th[n.w1 + (int64_t(co) * kK + ky) * kK + kx] * x[(yy + ky) * H + xx + kx];",
     "acc += th[n.w1 + (int64_t(co) * kK + (kK - 1 - ky)) * kK + (kK - 1 - kx)] * x[(yy + ky) * H + xx + kx];",
     "cnn"),
    ("conv2 reads the wrong input channel", "cnn_oracle.cpp",
     "a1[(size_t(ci) * P1 + yy + ky) * P1 + xx + kx];",
     "a1[(size_t((ci + 1) % n.c1) * P1 + yy + ky) * P1 + xx + kx];", "cnn"),
    # the schedules
    ("queue commits the latest-finishing worker", "schedule_oracle.cpp",
     "if (finish[w] < finish[best]) best = w;", "if (finish[w] > finish[best]) best = w;", "schedule"),
    ("uniform tick never picks the last worker", "schedule_oracle.cpp",
     "order[t] = int32_t((u32 * uint64_t(n)) >> 32);",
     "order[t] = int32_t((u32 * uint64_t(n - 1)) >> 32);", "schedule"),
]


def _build(tmp: Path, tag: str, edit=None) -> Path:
    d = tmp / tag
    d.mkdir()
    srcs = []
    for src in SOURCES:
        text = src.read_text()
        if edit and src.name == edit[0]:
            assert text.count(edit[1]) == 1, f"{tag}: the planted text must occur once in {src.name}"
            text = text.replace(edit[1], edit[2])
        (d / src.name).write_text(text)
        srcs.append(d / src.name)
    return compile_library(srcs, d / "liboracle.so")


def _pins_pass(lib: Path, pins: str) -> subprocess.CompletedProcess:
    env = dict(os.environ, ORACLE_LIBRARY=str(lib), OMP_NUM_THREADS="2")
    return subprocess.run([sys.executable, "-m", "pytest", PINS[pins], "-x", "-q", "-p", "no:cacheprovider",
                           "-m", "not gpu"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)


def test_unaltered_copy_passes_every_pin(tmp_path):
    lib = _build(tmp_path, "unaltered")
    for pins in PINS:
        r = _pins_pass(lib, pins)
        assert r.returncode == 0, (pins, r.stdout[-2000:])


def test_every_planted_mistake_fails_a_pin(tmp_path):
    def one(i_mistake):
        i, (name, src, old, new, pins) = i_mistake
        lib = _build(tmp_path, f"m{i}", (src, old, new))
        r = _pins_pass(lib, pins)
        return name, r.returncode, r.stdout[-600:]

    with ThreadPoolExecutor(max_workers=4) as ex:
        results = list(ex.map(one, enumerate(MISTAKES)))
    survived = [(name, out) for name, rc, out in results if rc == 0]
    assert not survived, f"planted mistakes the pins did not catch: {survived}"
    # a failing run must be a failing pin, not a crash of the harness
    for name, rc, out in results:
        assert rc == 1, (name, rc, out)
