"""Pin the CPU oracle to the paper and to definitions outside it (CPU only)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import workloads as W
from pins import (build, check_advance, check_apply, check_argmax, check_chain, check_golden,
                  check_masks, check_numbering, expected_row, prefix_ids, random_case, row_ids)


@pytest.mark.parametrize("name", ["appG1_worked_example.json", "fig2_alignment.json", "appH9_noncanonical.json",
                                  "sec42_prefix_values.json"])
def test_paper_worked_examples(oracle_lib, name):
    """App. G.1 Steps 1-4 (29 nodes, 44 chars, listed rows), Fig. 2's masks and
    App. H.9's canonical and non-canonical splits of one value."""
    check_golden(name)


@pytest.mark.parametrize("seed", range(40))
def test_numbering_closed_form(oracle_lib, seed):
    strings, _ = random_case(seed)
    check_numbering(strings)


@pytest.mark.parametrize("seed", range(60))
def test_masks_equal_prefix_enumeration(oracle_lib, seed):
    """Exhaustive over all (node, token): bit == [prefix(n)+v is a prefix of some e]."""
    strings, toks = random_case(1000 + seed)
    check_masks(strings, toks)


@pytest.mark.parametrize("seed", range(30))
def test_advance_matches_prefix_walk(oracle_lib, seed):
    strings, toks = random_case(2000 + seed)
    check_advance(strings, toks, seed)


@pytest.mark.parametrize("seed", range(15))
def test_apply_by_definition(oracle_lib, seed):
    strings, toks = random_case(3000 + seed)
    check_apply(strings, toks, seed)


def test_argmax_first_maximum(oracle_lib):
    check_argmax(7)


@pytest.mark.parametrize("s", [b"a", b"medical_billing", bytes([0, 255, 0, 255, 7])])
def test_single_string_chain(oracle_lib, s):
    check_chain(s)


def test_empty_string_makes_root_terminal(oracle_lib):
    toks = [b"a", b"ab", b""]
    t, voc = build([b"", b"ab"], toks)
    m = oracle.mask_all(t, voc)
    assert row_ids(m[0], 3) == {0, 1, 2}      # root: a, ab and EOS
    t2, voc2 = build([b""], toks)
    assert t2.num_nodes == 1
    assert row_ids(oracle.mask_all(t2, voc2)[0], 3) == {2}


def test_empty_set(oracle_lib):
    t, voc = build([], [b"a", b""])
    assert t.num_nodes == 1
    assert row_ids(oracle.mask_all(t, voc)[0], 2) == set()


# --------------------------------------------------------- invariants on a real-sized set

@pytest.fixture(scope="module")
def cfg1(oracle_lib):
    w = W.config(1)
    t = oracle.Trie(w.set_bytes, w.set_offsets)
    voc = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    m = oracle.mask_all(t, voc, nthreads=4)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    toks = W.unpack(w.vocab_bytes, w.vocab_offsets)
    ids, E = prefix_ids(strings)
    return w, t, voc, m, strings, toks, ids, E


def _allowed(m, n, v):
    return bool((m[n, v // 32] >> (v % 32)) & 1)


def test_cfg1_node_count(cfg1):
    w, t, voc, m, strings, toks, ids, E = cfg1
    assert t.num_nodes == len(ids)
    assert m.shape == (len(ids), (w.V + 31) // 32)


def test_invariant_tokenization_paths_allowed(cfg1):
    """Every step of the byte-by-byte and of the greedy longest-match
    tokenization of every e_i is allowed; EOS is allowed at its end (Sec. 5.3:
    100% validity; App. G.5 proof condition (i))."""
    w, t, voc, m, strings, toks, ids, E = cfg1
    tok_id = {tk: i for i, tk in enumerate(toks[:-1])}
    maxlen = max(len(x) for x in toks)
    for s in strings:
        for greedy in (False, True):
            p, n = 0, 0
            while p < len(s):
                L = 1
                if greedy:
                    L = max(L_ for L_ in range(1, min(maxlen, len(s) - p) + 1)
                            if s[p:p + L_] in tok_id)
                v = tok_id[s[p:p + L]]
                assert _allowed(m, n, v)
                n = ids[s[:p + L]]
                p += L
            assert _allowed(m, n, w.V - 1)


def test_invariant_leaves_only_eos(cfg1):
    w, t, voc, m, strings, toks, ids, E = cfg1
    has_child = np.zeros(t.num_nodes, bool)
    has_child[t.parent[1:]] = True
    leaves = np.nonzero(~has_child)[0]
    assert len(leaves) > 0
    for n in leaves:
        assert t.terminal[n]
        assert row_ids(m[n], w.V) == {w.V - 1}


def test_invariant_eos_iff_terminal_and_padding(cfg1):
    w, t, voc, m, strings, toks, ids, E = cfg1
    eos = w.V - 1
    eos_bits = (m[:, eos // 32] >> (eos % 32)) & 1
    assert np.array_equal(eos_bits.astype(bool), t.terminal.astype(bool))
    tail = m[:, -1] >> np.uint32((eos % 32) + 1) if eos % 32 != 31 else np.zeros(1, np.uint32)
    assert not np.any(tail)


def test_invariant_rows_nonempty(cfg1):
    """All 256 single bytes are tokens, so every node has a continuation or EOS."""
    w, t, voc, m, *_ = cfg1
    assert np.all(m.any(axis=1))


def test_invariant_prefix_closure(cfg1):
    """v = u.w allowed at n  =>  u allowed at n and w allowed at delta*(n, u)."""
    w, t, voc, m, strings, toks, ids, E = cfg1
    tok_id = {tk: i for i, tk in enumerate(toks[:-1])}
    inv = {i: p for p, i in ids.items()}
    checked = 0
    for n in range(0, t.num_nodes, 7):
        for v in row_ids(m[n], w.V):
            if v == w.V - 1:
                continue
            tv = toks[v]
            for cut in range(1, len(tv)):
                u, x = tv[:cut], tv[cut:]
                if u in tok_id and x in tok_id:
                    assert _allowed(m, n, tok_id[u])
                    assert _allowed(m, ids[inv[n] + u], tok_id[x])
                    checked += 1
    assert checked > 0


def test_invariant_equal_suffix_languages_equal_rows(cfg1):
    """Nodes whose remaining languages {s : prefix(n)+s in E} coincide have the
    same row (Myhill-Nerode classes, Prop. 1)."""
    w, t, voc, m, strings, toks, ids, E = cfg1
    inv = {i: p for p, i in ids.items()}
    lang: dict[frozenset, list[int]] = {}
    for n in range(t.num_nodes):
        p = inv[n]
        key = frozenset(s[len(p):] for s in E if s.startswith(p))
        lang.setdefault(key, []).append(n)
    groups = [g for g in lang.values() if len(g) > 1]
    assert groups
    for g in groups:
        for n in g[1:]:
            assert np.array_equal(m[n], m[g[0]])


def test_invariant_advance_lands_on_prefix_node(cfg1):
    """delta*(root, concatenated token bytes) = node of that prefix."""
    w, t, voc, m, strings, toks, ids, E = cfg1
    tok_id = {tk: i for i, tk in enumerate(toks[:-1])}
    r = np.random.default_rng(0)
    for s in strings[:50]:
        cuts = sorted(set(r.integers(1, len(s), 3).tolist()))
        pieces = [s[a:b] for a, b in zip([0] + cuts, cuts + [len(s)])]
        pieces = [[bytes([c]) for c in pc] if pc not in tok_id else [pc] for pc in pieces]
        seq = [tok_id[x] for pc in pieces for x in pc]
        st = np.zeros(1, np.int32)
        acc = b""
        for v in seq:
            st, e = oracle.advance(t, voc, st, np.array([v], np.int32))
            acc += toks[v]
            assert e == 0 and st[0] == ids[acc]
        st, e = oracle.advance(t, voc, st, np.array([w.V - 1], np.int32))
        assert st[0] == oracle.FINISHED


def test_invariant_greedy_decode_always_valid(cfg1):
    """Greedy decoding under the masks emits only set members (100% validity)."""
    w, t, voc, m, strings, toks, ids, E = cfg1
    B, steps = 16, 40
    r = np.random.default_rng(1)
    lg = [(r.standard_normal((B, w.V)).astype(np.float32)).view(np.uint32) for _ in range(steps)]
    masked, tks, sts, errors = oracle.decode(t, voc, lg, np.zeros(B, np.int32))
    assert errors == 0
    out = [b""] * B
    done = [False] * B
    for k in range(steps):
        for b in range(B):
            if not done[b]:
                if tks[k][b] == w.V - 1:
                    done[b] = True
                else:
                    out[b] += toks[tks[k][b]]
    assert all(done)
    assert all(o in E for o in out)


def test_cfg3_sampled_rows_match_enumeration(oracle_lib):
    """Full-size code set and 152K vocab: sampled rows against the prefix set."""
    w = W.config(3)
    t = oracle.Trie(w.set_bytes, w.set_offsets)
    voc = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    toks = W.unpack(w.vocab_bytes, w.vocab_offsets)
    ids, E = prefix_ids(strings)
    inv = {i: p for p, i in ids.items()}
    assert t.num_nodes == len(ids)
    rows = [0, 1, 5, 27, 300, len(ids) // 2, len(ids) - 1]
    m = oracle.mask_rows(t, voc, rows)
    for k, n in enumerate(rows):
        assert row_ids(m[k], w.V) == expected_row(inv[n], toks, ids, E)
