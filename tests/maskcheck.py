"""Whole-mask comparison against a list of expected set bits.

A dense mask too large to rebuild on the host (the 256-request forest: 4.8 M
rows of 4,000 words, 76 GB) is compared with the oracle's sparse result, the
(row, token) pairs of every allowed move (``oracle.AhoCorasick.pairs`` plus EOS
at terminal nodes). The expected words are assembled chunk by chunk on the
mask's own device with plain torch indexing: every pair adds 2^(token % 32)
to word token // 32 of its row. The pairs of one word are distinct, so their
sum is their bitwise OR. The mask's words, read as unsigned 32-bit values,
must equal those sums everywhere, so a missing bit, an extra bit and a bit in
the wrong row or word all fail.
"""
from __future__ import annotations

import numpy as np


def assert_mask_equals_pairs(mask, rows: np.ndarray, tokens: np.ndarray,
                             chunk_words: int = 1 << 28) -> None:
    """Assert that ``mask`` ([N, W] int32 tensor, any device) has a set bit at
    exactly the given (row, token) pairs. ``chunk_words`` bounds the words
    compared at once (two int64 temporaries of that many words)."""
    import torch
    N, Wd = mask.shape
    rows = np.asarray(rows, dtype=np.int64)
    tokens = np.asarray(tokens, dtype=np.int64)
    assert rows.shape == tokens.shape
    order = np.lexsort((tokens, rows))
    rows, tokens = rows[order], tokens[order]
    if rows.size:
        assert rows[0] >= 0 and rows[-1] < N, "pair row out of range"
        assert tokens.min() >= 0 and tokens.max() < 32 * Wd, "pair token out of range"
        assert not np.any((rows[1:] == rows[:-1]) & (tokens[1:] == tokens[:-1])), "repeated pair"
    dev = mask.device
    step = max(1, chunk_words // Wd)
    for r0 in range(0, N, step):
        r1 = min(N, r0 + step)
        a, b = np.searchsorted(rows, [r0, r1])
        want = torch.zeros((r1 - r0) * Wd, dtype=torch.int64, device=dev)
        if b > a:
            rr = torch.as_tensor(rows[a:b] - r0, device=dev)
            tt = torch.as_tensor(tokens[a:b], device=dev)
            want.index_put_((rr * Wd + torch.div(tt, 32, rounding_mode="floor"),),
                            torch.ones_like(tt) << (tt % 32), accumulate=True)
        got = mask[r0:r1].reshape(-1).to(torch.int64)
        got &= 0xFFFFFFFF
        if not torch.equal(got, want):
            k = int((got != want).nonzero()[0].item())
            raise AssertionError(f"row {r0 + k // Wd}, word {k % Wd}: mask {int(got[k]):#010x}, "
                                 f"expected {int(want[k]):#010x}")
        del want, got


def forest_pairs(ac, strings: list[bytes], set_index, roots, V: int, nthreads: int = 1):
    """Every allowed (row, token) pair of a forest, from the oracle: per set,
    the Aho-Corasick pairs of the set's own trie and EOS (token V - 1) at its
    terminal nodes, with the set's node ids offset by its root."""
    import oracle
    from paper_2608_12574_gb300 import workloads as W
    parts_r, parts_t = [], []
    for i in range(len(set_index) - 1):
        ot = oracle.Trie(*W.pack(strings[set_index[i]:set_index[i + 1]]))
        r, t = ac.pairs(ot, nthreads=nthreads)
        term = np.nonzero(ot.terminal)[0]
        parts_r += [r.astype(np.int64) + int(roots[i]), term.astype(np.int64) + int(roots[i])]
        parts_t += [t.astype(np.int64), np.full(len(term), V - 1, np.int64)]
    if not parts_r:
        return np.zeros(0, np.int64), np.zeros(0, np.int64)
    return np.concatenate(parts_r), np.concatenate(parts_t)
