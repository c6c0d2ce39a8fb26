"""Pins of the oracle's character-position masks for fixed formats (App. K).

The format's language is the finite product of its byte classes, so the
prefix-set definition that pins the trie oracle (App. G.5 conditions, see
pins.py) pins the position automaton as well: row p must equal the row of
every prefix of length p. Plus a closed form (all classes full) and a date
format worked by hand.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import workloads as W
from pins import (check_fmt_advance, check_fmt_closed_form, check_fmt_masks, fmt_bitmaps, fmt_case,
                  row_ids)


@pytest.mark.parametrize("seed", range(60))
def test_fmt_masks_equal_prefix_enumeration(oracle_lib, seed):
    cls, toks = fmt_case(7000 + seed)
    check_fmt_masks(cls, toks)


@pytest.mark.parametrize("seed", range(30))
def test_fmt_advance_matches_prefix_walk(oracle_lib, seed):
    cls, toks = fmt_case(7100 + seed)
    check_fmt_advance(cls, toks, seed)


@pytest.mark.parametrize("L", [0, 1, 4, 9])
def test_fmt_closed_form_full_classes(oracle_lib, L):
    check_fmt_closed_form(L, [b"a", b"ab", b"abcdef", b"", b"\x00\xff", b"0123456789", b"q"])


def test_fmt_date_worked_by_hand(oracle_lib):
    """YYYY-MM-DD: digits everywhere but '-' at positions 4 and 7."""
    digits = list(range(0x30, 0x3A))
    cls = [digits] * 4 + [[0x2D]] + [digits] * 2 + [[0x2D]] + [digits] * 2
    toks = [b"2024", b"-", b"20", b"24-", b"-0", b"12", b"1", b"a", b"2024-12-01", b"-12-", b"", b""]
    f = oracle.Format(fmt_bitmaps(cls))
    voc = oracle.Vocab(*W.pack(toks))
    V = len(toks)
    m = f.mask_all(voc)
    name = {i: t for i, t in enumerate(toks)}
    rows = {p: sorted(name[v] for v in row_ids(m[p], V) if v != V - 1) for p in range(11)}
    assert rows[0] == sorted([b"2024", b"20", b"12", b"1", b"2024-12-01"])
    assert rows[2] == sorted([b"20", b"24-", b"12", b"1"])
    assert rows[4] == sorted([b"-", b"-0", b"-12-"])
    assert rows[5] == sorted([b"20", b"24-", b"12", b"1"])   # 5, 6 digits, 7 the dash
    assert rows[8] == sorted([b"20", b"12", b"1"])
    assert rows[9] == [b"1"]
    assert rows[10] == [] and row_ids(m[10], V) == {V - 1}
    assert all(V - 1 not in row_ids(m[p], V) for p in range(10))
    # 2024 | -12- | 01 | EOS
    st, err = f.advance(voc, np.zeros(1, np.int32), np.array([0], np.int32))
    assert st.tolist() == [4]
    st, _ = f.advance(voc, st, np.array([9], np.int32))
    assert st.tolist() == [8]
    st, _ = f.advance(voc, st, np.array([5], np.int32))   # "12" fills the day
    assert st.tolist() == [10]
    st, _ = f.advance(voc, st, np.array([V - 1], np.int32))
    assert st.tolist() == [oracle.FINISHED] and err == 0
