"""The paper's Aho-Corasick precomputation (oracle/ac.c) against the brute-force
oracle: the same masks, on small random sets (every node, every token) and on
the K=100 and K=10,000 workloads (CPU only)."""
from __future__ import annotations

import os

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import workloads as W
from pins import build, random_case

NCPU = os.cpu_count() or 1


@pytest.mark.parametrize("seed", range(40))
def test_ac_equals_oracle_small(oracle_lib, seed):
    strings, toks = random_case(1000 + seed)
    t, voc = build(strings, toks)
    ac = oracle.AhoCorasick(voc)
    assert np.array_equal(ac.mask(t), oracle.mask_all(t, voc))


def test_ac_worked_example(oracle_lib):
    """App. G.1: the automaton over {medical, _bill, _cod, _rec, ing, ords}
    attributes _bill/_cod/_rec to the node after 'medical'."""
    strings = [b"medical_billing", b"medical_coding", b"medical_records"]
    toks = [b"medical", b"_bill", b"_cod", b"_rec", b"ing", b"ords", b""]
    t, voc = build(strings, toks)
    rows, tk = oracle.AhoCorasick(voc).pairs(t)
    n7 = [i for i in range(t.num_nodes) if t.prefix(i) == b"medical"][0]
    assert sorted(tk[rows == n7].tolist()) == [1, 2, 3]
    assert tk[rows == 0].tolist() == [0]


@pytest.mark.parametrize("cfg", [1, 3])
def test_ac_equals_oracle_configs(oracle_lib, cfg):
    w = W.config(cfg)
    t = oracle.Trie(w.set_bytes, w.set_offsets)
    voc = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    ac = oracle.AhoCorasick(voc)
    got = ac.mask(t, nthreads=NCPU)
    step = 2048
    for r0 in range(0, t.num_nodes, step):
        rows = np.arange(r0, min(r0 + step, t.num_nodes), dtype=np.int32)
        assert np.array_equal(got[r0:r0 + len(rows)], oracle.mask_rows(t, voc, rows, nthreads=NCPU)), r0


def test_ac_forest_roots(oracle_lib):
    """Trees concatenated with parent -1 at each root (the forest layout)."""
    w = W.dynamic_requests(3)
    voc = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    ac = oracle.AhoCorasick(voc)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    for i in range(3):
        st = strings[w.set_index[i]:w.set_index[i + 1]]
        t = oracle.Trie(*W.pack(st))
        rows = np.arange(0, t.num_nodes, 97, dtype=np.int32)
        assert np.array_equal(ac.mask(t, nthreads=NCPU)[rows], oracle.mask_rows(t, voc, rows, nthreads=NCPU))
