"""The whole-mask comparison used for the 256-request forest, checked on CPU.

``maskcheck.assert_mask_equals_pairs`` compares a dense mask with the
oracle's sparse pairs. Here the dense mask is the brute-force oracle's own
(``oracle.mask_all``), so the comparison must pass, and every planted change
of one bit (cleared, added, the sign bit, moved to the next row or word) must
fail, also when the rows are compared in small chunks with a ragged last one.
``maskcheck.forest_pairs`` is checked the same way on a forest whose roots
come from the host builder.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from maskcheck import assert_mask_equals_pairs, forest_pairs
from paper_2608_12574_gb300 import workloads as W
from pins import random_case


@pytest.fixture(scope="module")
def k100(oracle_lib):
    w = W.config(1)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    dense = oracle.mask_all(ot, ov, nthreads=4)
    ac = oracle.AhoCorasick(ov)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    rows, toks = forest_pairs(ac, strings, [0, len(strings)], [0], w.V)
    return dense, rows, toks


def _t(a: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int32))


@pytest.mark.parametrize("chunk", [1 << 28, 3 * 1000 + 7, 1000])
def test_oracle_mask_equals_its_pairs(k100, chunk):
    dense, rows, toks = k100
    assert dense.shape == (1384, 1000)
    assert int(np.unpackbits(dense.view(np.uint8)).sum()) == rows.size
    assert_mask_equals_pairs(_t(dense), rows, toks, chunk_words=chunk)


def _flip(dense: np.ndarray, row: int, token: int) -> np.ndarray:
    d = dense.copy()
    d[row, token // 32] ^= np.uint32(1) << np.uint32(token % 32)
    return d


@pytest.mark.parametrize("chunk", [1 << 28, 3 * 1000 + 7])
def test_planted_bit_changes_fail(k100, chunk):
    dense, rows, toks = k100
    i = int(np.nonzero(rows < 1383)[0][len(rows) // 3])
    r, t = int(rows[i]), int(toks[i])                   # an allowed pair, not in the last row
    cases = {
        "cleared": _flip(dense, r, t),
        "flipped in the last row": _flip(dense, 1383, 31_998),
        "sign bit": _flip(dense, 700, 32 * 17 + 31),
        "moved to the next row": _flip(_flip(dense, r, t), r + 1, t),
        "moved to the next word": _flip(_flip(dense, r, t), r, (t + 32) % 32_000),
    }
    for name, bad in cases.items():
        assert not np.array_equal(bad, dense), name
        with pytest.raises(AssertionError):
            assert_mask_equals_pairs(_t(bad), rows, toks, chunk_words=chunk)


def test_forest_pairs_match_the_forest_layout(oracle_lib):
    from paper_2608_12574_gb300 import triemask as T
    from paper_2608_12574_gb300 import _build
    _build.build()
    _, toks = random_case(7)
    toks = [t for t in toks[:-1] if t] + [b""]                  # EOS last
    sets = [random_case(s)[0] for s in (1, 2, 3, 4, 11)]
    strings = [s for st in sets for s in st]
    index = np.cumsum([0] + [len(st) for st in sets]).astype(np.int32)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h = T.trie_build_many(sb, so, index)
    roots = h.roots()
    ov = oracle.Vocab(vb, vo)
    parts = [oracle.mask_all(oracle.Trie(*W.pack(st)), ov) for st in sets]
    dense = np.concatenate(parts)
    assert dense.shape[0] == h.num_nodes
    assert list(roots) == list(np.cumsum([0] + [p.shape[0] for p in parts[:-1]]))
    rows, tk = forest_pairs(oracle.AhoCorasick(ov), strings, index, roots, len(toks))
    for chunk in (1 << 20, dense.shape[1] * 2 + 1):
        assert_mask_equals_pairs(_t(dense), rows, tk, chunk_words=chunk)
    with pytest.raises(AssertionError):                          # a set's pairs at another set's root
        shifted = list(roots[:-1]) + [int(roots[-1]) - 1]
        r2, t2 = forest_pairs(oracle.AhoCorasick(ov), strings, index, shifted, len(toks))
        assert_mask_equals_pairs(_t(dense), r2, t2)
    h.destroy()
