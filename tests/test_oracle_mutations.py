"""Plant plausible mistakes in a copy of the oracle and check the pins catch each.

Every mutant is a textual edit of oracle/oracle.c, compiled into a temporary
directory (CPU only) and checked in a child process, so that only an
AssertionError from a pin counts as caught. A mutant that passes all pins
would mean the pins cannot tell that mistake from the correct oracle.
"""
from __future__ import annotations

import os
import subprocess
import sys

import pytest

import oracle
from pins import (check_advance, check_apply, check_argmax, check_chain, check_fmt_advance,
                  check_fmt_closed_form, check_fmt_masks, check_golden, check_masks, check_numbering,
                  fmt_case, random_case)

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTANTS = {
    "overshoot_allowed": ("        if (x < 0) return -1;\n    }\n    return x;",
                          "        if (x < 0) return n;\n    }\n    return x;"),
    "empty_token_allowed": ("if (e <= a) return -1;", "if (e <= a) return n;"),
    "eos_ignores_terminal": ("if (!node || t->terminal[n]) row", "if (!node) row"),
    "eos_everywhere": ("if (!node || t->terminal[n]) row", "if (1) row"),
    "bit_index_off_by_one": ("if (walk(t, n, vb, vo, v) >= 0) row[v / 32] |= 1u << (v % 32);",
                             "if (walk(t, n, vb, vo, v) >= 0) row[v / 32] |= 1u << ((v + 1) % 32);"),
    "last_token_skipped": ("for (int32_t v = 0; v < eos; v++)", "for (int32_t v = 0; v < eos - 1; v++)"),
    "siblings_descending": ("        for (int b = 0; b < 256; b++)\n            if (ch[(int64_t)x * 256 + b] >= 0) order",
                            "        for (int b = 255; b >= 0; b--)\n            if (ch[(int64_t)x * 256 + b] >= 0) order"),
    "insertion_order_numbering": ("for (int64_t i = 0; i < n; i++) newid[order[i]] = (int32_t)i;",
                                  "for (int64_t i = 0; i < n; i++) { order[i] = (int32_t)i; newid[i] = (int32_t)i; }"),
    "finished_eos_dies": ("nxt = (v == eos) ? ORACLE_FINISHED : ORACLE_DEAD;",
                          "nxt = ORACLE_DEAD;"),
    "eos_finishes_anywhere": ("nxt = t->terminal[s] ? ORACLE_FINISHED : ORACLE_DEAD;",
                              "nxt = ORACLE_FINISHED;"),
    "dead_moves_not_counted": ("if (nxt == ORACLE_DEAD) errors++;", "if (0) errors++;"),
    "bf16_neg_inf_wrong": ("= 0xFF80u;", "= 0x7F80u;"),
    "f32_neg_inf_wrong": ("= 0xFF800000u;", "= 0xFF000000u;"),
    "argmax_last_tie": ("if (v == 0 || x > bv)", "if (v == 0 || x >= bv)"),
    "fmt_length_bound_off_by_one": ("if (len < 1 || len > (int64_t)(L - p)) return 0;",
                                    "if (len < 1 || len > (int64_t)(L - p + 1)) return 0;"),
    "fmt_class_of_token_position": ("if (!fmt_class_has(classes, p + (int32_t)i, vb[vo[v] + i])) return 0;",
                                    "if (!fmt_class_has(classes, (int32_t)i, vb[vo[v] + i])) return 0;"),
    "fmt_eos_anywhere": ("if (v == V - 1) return p == L;", "if (v == V - 1) return 1;"),
    "fmt_advance_one_position": ("s + (int32_t)(vo[v + 1] - vo[v])", "s + 1"),
    "terminal_not_marked_for_prefix_values": ("        term[x] = 1;\n", "        if (x > 0 || offsets[i+1] > offsets[i]) term[x] = 1;\n        if (ch[x * 256 + 0] >= 0) term[x] = 0;\n"),
}


def _all_pins():
    check_golden("appG1_worked_example.json")
    check_golden("fig2_alignment.json")
    check_golden("appH9_noncanonical.json")
    check_golden("sec42_prefix_values.json")
    check_argmax(7)
    check_chain(b"medical_billing")
    check_chain(bytes([0, 255, 0, 255, 7]))
    for seed in range(40):
        strings, toks = random_case(1000 + seed)
        check_numbering(strings)
        check_masks(strings, toks)
        check_advance(strings, toks, seed)
        check_apply(strings, toks, seed)
    for seed in range(30):
        cls, ftoks = fmt_case(7000 + seed)
        check_fmt_masks(cls, ftoks)
        check_fmt_advance(cls, ftoks, seed)
    check_fmt_closed_form(5, [b"a", b"ab", b"abcdef", b"", b"xyz", b"\x00\xff", b""])


TESTS = os.path.dirname(os.path.abspath(__file__))
CHILD = """
import sys
sys.path[:0] = [{root!r}, {tests!r}]
import oracle, test_oracle_mutations as m
with oracle.use_library({lib!r}):
    try:
        m._all_pins()
    except AssertionError:
        print("PIN-FAILED")
        sys.exit(3)
print("PINS-PASSED")
"""


def _run_pins_with(lib: str) -> subprocess.CompletedProcess:
    code = CHILD.format(root=os.path.dirname(TESTS), tests=TESTS, lib=lib)
    return subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300)


def _compile(src_text: str, tmp_path, name: str) -> str:
    path = tmp_path / f"{name}.c"
    path.write_text(src_text)
    lib = tmp_path / f"lib{name}.so"
    subprocess.check_call(["gcc", "-O1", "-shared", "-fPIC", "-std=c99", "-o", str(lib), str(path)])
    return str(lib)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(oracle_lib, tmp_path, name):
    src = open(SRC).read()
    old, new = MUTANTS[name]
    assert src.count(old) == 1, f"mutation site for {name} not unique / not found"
    r = _run_pins_with(_compile(src.replace(old, new), tmp_path, "mut"))
    assert r.returncode == 3 and "PIN-FAILED" in r.stdout, (r.returncode, r.stdout[-500:], r.stderr[-2000:])


def test_unmutated_copy_passes(oracle_lib, tmp_path):
    r = _run_pins_with(_compile(open(SRC).read(), tmp_path, "same"))
    assert r.returncode == 0 and "PINS-PASSED" in r.stdout, (r.stdout[-500:], r.stderr[-2000:])
