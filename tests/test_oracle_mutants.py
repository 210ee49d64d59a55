"""The oracle's pins catch plausible mistakes: each case below plants one mistake in a copy
of oracle/hs_oracle.c (on the CPU), builds it, and runs tests/test_oracle_pins.py against
it in a child process; at least one pin must fail for every mutant, and the unmodified copy
built the same way must pass them all."""
import os
import subprocess
import sys

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "hs_oracle.c")

UPDATE = "S[i * d_v + j] = g * S[i * d_v + j] + ki * bf16_to_double(vt[j]);"
OUTPUT = "acc += bf16_to_double(qt[i]) * S[i * d_v + j];"
UPDATE_BLOCK_START = "        /* S_t = diag(g_t) S_{t-1} + k_t v_t^T */"
OUTPUT_BLOCK_START = "        /* o_t = q_t S_t */"
CKPT_BLOCK_START = "        /* checkpoint: the state of prefix"


def _output_before_update(src: str) -> str:
    """o_t from S_{t-1}: the output block moved in front of the update."""
    a = src.index(UPDATE_BLOCK_START)
    b = src.index(OUTPUT_BLOCK_START)
    c = src.index(CKPT_BLOCK_START)
    return src[:a] + src[b:c] + src[a:b] + src[c:]


MUTANTS = {
    "dropped k v^T": lambda s: s.replace(UPDATE, "S[i * d_v + j] = g * S[i * d_v + j];"),
    "gate not exponentiated": lambda s: s.replace("double g = exp((double)at[i]);",
                                                  "double g = (double)at[i];"),
    "gate of the value column": lambda s: s.replace(
        UPDATE, "S[i * d_v + j] = exp((double)at[j]) * S[i * d_v + j] + ki * bf16_to_double(vt[j]);"),
    "transposed state in the output": lambda s: s.replace(
        OUTPUT, "acc += bf16_to_double(qt[i]) * S[j * d_v + i];"),
    "output sign": lambda s: s.replace(OUTPUT, "acc -= bf16_to_double(qt[i]) * S[i * d_v + j];"),
    "output from the state before the token": _output_before_update,
    "checkpoint one token early": lambda s: s.replace("(pos0 + t + 1) % C == 0", "(pos0 + t) % C == 0"),
    "alignment on the full prompt": lambda s: s.replace("for (int64_t b = N - 1; b >= 0; --b)",
                                                        "for (int64_t b = N; b >= 0; --b)"),
    "alignment ignores the hit": lambda s: s.replace("if (b > hit_len)\n            continue;", ""),
    "bf16 widened from the wrong bits": lambda s: s.replace("((uint32_t)b) << 16", "((uint32_t)b) << 15"),
    "state bytes counted in bf16": lambda s: s.replace("n_heads * d_k * d_v * 4", "n_heads * d_k * d_v * 2"),
    "state bytes without the heads": lambda s: s.replace("n_lin_layers * n_heads * d_k * d_v * 4",
                                                         "n_lin_layers * d_k * d_v * 4"),
    "scatter to the staging index": lambda s: s.replace(
        "memcpy(cache[l] + (int64_t)bt[j] * page_bytes,", "memcpy(cache[l] + (int64_t)j * page_bytes,"),
    "gather from the staging index": lambda s: s.replace(
        "cache[l] + (int64_t)bt[j] * page_bytes, (size_t)page_bytes);",
        "cache[l] + (int64_t)j * page_bytes, (size_t)page_bytes);"),
    "gather one page short": lambda s: s.replace(
        "j < n_pages; ++j)\n            memcpy(staging", "j < n_pages - 1; ++j)\n            memcpy(staging"),
    "slice ignores the column offset": lambda s: s.replace("+ r * row_bytes + col_off;", "+ r * row_bytes;"),
    "slice of the first row only": lambda s: s.replace("+ r * row_bytes + col_off;", "+ col_off;"),
    "slice direction swapped": lambda s: s.replace("if (gather)\n                    memcpy(s, c,",
                                                   "if (!gather)\n                    memcpy(s, c,"),
    "state copy from the first slot": lambda s: s.replace("memcpy(dst[i], src[i],", "memcpy(dst[i], src[0],"),
    "state copy in reverse slot order": lambda s: s.replace("memcpy(dst[i], src[i],",
                                                            "memcpy(dst[i], src[n - 1 - i],"),
    "state copy of floats_each bytes": lambda s: s.replace("(size_t)floats_each * sizeof(float)",
                                                           "(size_t)floats_each"),
}


def _run_pins(lib_path: str) -> subprocess.CompletedProcess:
    env = dict(os.environ, HS_ORACLE_LIB=lib_path)
    return subprocess.run([sys.executable, "-m", "pytest", os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                           "-x", "-q", "-p", "no:cacheprovider"],
                          cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)


def _build(tmp_path, name: str, src: str) -> str:
    c = tmp_path / f"{name}.c"
    c.write_text(src)
    so = tmp_path / f"lib{name}.so"
    oracle.compile_to(str(c), str(so))
    return str(so)


def test_unmodified_copy_passes_the_pins(tmp_path):
    r = _run_pins(_build(tmp_path, "orig", open(SRC).read()))
    assert r.returncode == 0, r.stdout[-2000:]


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_each_planted_mistake_fails_a_pin(tmp_path, name):
    src = open(SRC).read()
    mutated = MUTANTS[name](src)
    assert mutated != src, f"mutation {name!r} did not apply"
    r = _run_pins(_build(tmp_path, "mutant", mutated))
    # 1 = some test failed (0 would mean every pin passed; >1 an error of the harness)
    assert r.returncode == 1, (name, r.returncode, r.stdout[-2000:])
