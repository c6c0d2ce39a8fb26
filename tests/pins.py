"""Checks that pin the CPU oracle to facts fixed outside it.

Each ``check_*`` raises AssertionError on a mismatch. They are used by
``test_oracle_pins.py`` on the real oracle and by ``test_oracle_mutations.py``
on copies of the oracle with planted mistakes.

The reference values are computed here from definitions, never from the
oracle:

* node ids: breadth-first order with siblings by ascending byte is the order
  of the distinct prefixes sorted by (length, bytes);
* mask bits: App. G.5 proof, conditions (i)+(ii): v is allowed at the node for
  prefix p iff p + bytes(v) is a prefix of some set string (the hash-set of
  prefixes, as in the hash-set prefix matching of App. H.10), plus EOS iff p is in the set;
* transitions: the same prefix set, with FINISHED / DEAD as the oracle header
  states them.
"""
from __future__ import annotations

import json
import os
import random

import numpy as np

import oracle
from paper_2608_12574_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
NEG_INF_F32 = 0xFF800000
NEG_INF_BF16 = 0xFF80


# ------------------------------------------------------------ definitions

def prefix_ids(strings: list[bytes]) -> tuple[dict[bytes, int], set[bytes]]:
    """Closed-form node numbering: distinct prefixes sorted by (len, bytes)."""
    P = {s[:j] for s in strings for j in range(len(s) + 1)}
    P.add(b"")
    order = sorted(P, key=lambda s: (len(s), s))
    return {p: i for i, p in enumerate(order)}, set(strings)


def expected_row(p: bytes, toks: list[bytes], ids: dict[bytes, int], E: set[bytes]) -> set[int]:
    eos = len(toks) - 1
    row = {v for v in range(eos) if toks[v] and (p + toks[v]) in ids}
    if p in E:
        row.add(eos)
    return row


def row_ids(words: np.ndarray, V: int) -> set[int]:
    bits = np.unpackbits(words.astype("<u4").view(np.uint8), bitorder="little")
    return set(np.nonzero(bits)[0].tolist())


def expected_next(p: bytes | None, state: int, tok: int, toks: list[bytes],
                  ids: dict[bytes, int], E: set[bytes]) -> int:
    eos = len(toks) - 1
    if state == oracle.DEAD:
        return oracle.DEAD
    if tok < 0 or tok >= len(toks):
        return oracle.DEAD
    if state == oracle.FINISHED:
        return oracle.FINISHED if tok == eos else oracle.DEAD
    if p is None:
        return oracle.DEAD
    if tok == eos:
        return oracle.FINISHED if p in E else oracle.DEAD
    if not toks[tok]:
        return oracle.DEAD
    q = p + toks[tok]
    return ids.get(q, oracle.DEAD)


# ------------------------------------------------------------ small random inputs

def random_case(seed: int):
    """A small set and vocab over a 2-4 byte alphabet: duplicates, prefixes of
    other strings, the empty string, bytes 0x00 / 0xFF, byte-less tokens."""
    r = random.Random(seed)
    alpha = r.sample([0, 1, 0x41, 0x5F, 0x7A, 0x80, 0xFF], r.randint(2, 4))
    K = r.randint(1, 20)
    strings = [bytes(r.choice(alpha) for _ in range(r.randint(0 if r.random() < 0.1 else 1, 7)))
               for _ in range(K)]
    if r.random() < 0.5 and strings:                  # a proper prefix of another value
        s = strings[r.randrange(len(strings))]
        strings.append(s[: r.randint(0, len(s))])
    if r.random() < 0.3:                              # duplicates
        strings += strings[: r.randint(1, len(strings))]
    V = r.randint(2, 300)
    toks = []
    for _ in range(V - 1):
        L = r.choice([0, 1, 1, 2, 2, 3, 4, 5])
        pool = alpha + ([r.randrange(256)] if r.random() < 0.2 else [])
        toks.append(bytes(r.choice(pool) for _ in range(L)))
    toks.append(b"")  # EOS
    return strings, toks


def build(strings: list[bytes], toks: list[bytes]):
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    return oracle.Trie(sb, so), oracle.Vocab(vb, vo)


# ------------------------------------------------------------ checks

def check_numbering(strings: list[bytes]) -> None:
    t, _ = build(strings, [b"a", b""])
    ids, E = prefix_ids(strings)
    assert t.num_nodes == len(ids), (t.num_nodes, len(ids))
    assert t.num_chars == sum(len(s) for s in E)
    for p, i in ids.items():
        assert t.prefix(i) == p, (i, t.prefix(i), p)
        assert bool(t.terminal[i]) == (p in E)
        assert t.depth[i] == len(p)
        if i:
            assert t.parent[i] == ids[p[:-1]] and t.label[i] == p[-1]


def check_masks(strings: list[bytes], toks: list[bytes]) -> None:
    t, voc = build(strings, toks)
    ids, E = prefix_ids(strings)
    V = len(toks)
    m = oracle.mask_all(t, voc)
    assert m.shape == (len(ids), (V + 31) // 32)
    for p, i in ids.items():
        got = row_ids(m[i], V)
        assert all(v < V for v in got), "padding bits set"
        assert got == expected_row(p, toks, ids, E), (p, sorted(got))
    # FINISHED / DEAD rows: EOS only
    m2 = oracle.mask_rows(t, voc, [oracle.FINISHED, oracle.DEAD])
    for k in range(2):
        assert row_ids(m2[k], V) == {V - 1}


def check_advance(strings: list[bytes], toks: list[bytes], seed: int) -> None:
    t, voc = build(strings, toks)
    ids, E = prefix_ids(strings)
    inv = {i: p for p, i in ids.items()}
    r = random.Random(seed)
    V = len(toks)
    B = 400
    states = np.array([r.choice([oracle.DEAD, oracle.FINISHED, len(ids), r.randrange(len(ids)),
                                 r.randrange(len(ids))]) for _ in range(B)], np.int32)
    tokens = np.array([r.choice([-1, V, V - 1, r.randrange(V), r.randrange(V)]) for _ in range(B)],
                      np.int32)
    got, err = oracle.advance(t, voc, states, tokens)
    want = [expected_next(inv.get(int(s)), int(s), int(v), toks, ids, E)
            for s, v in zip(states, tokens)]
    assert got.tolist() == want, [(int(s), int(v), g, w) for s, v, g, w in
                                  zip(states, tokens, got, want) if g != w][:5]
    want_err = sum(1 for s, w in zip(states, want) if w == oracle.DEAD and s != oracle.DEAD)
    assert err == want_err, (err, want_err)


def check_apply(strings: list[bytes], toks: list[bytes], seed: int) -> None:
    t, voc = build(strings, toks)
    ids, E = prefix_ids(strings)
    inv = {i: p for p, i in ids.items()}
    r = np.random.default_rng(seed)
    V = len(toks)
    B = 8
    states = r.choice(np.array([oracle.DEAD, oracle.FINISHED] + list(range(len(ids))), np.int32), B)
    for dtype, neg in ((np.uint32, NEG_INF_F32), (np.uint16, NEG_INF_BF16)):
        x = r.integers(0, np.iinfo(dtype).max, (B, V), dtype=dtype, endpoint=True)
        y = oracle.apply(t, voc, x, states)
        for b in range(B):
            s = int(states[b])
            allowed = expected_row(inv[s], toks, ids, E) if s >= 0 else {V - 1}
            keep = np.zeros(V, bool)
            keep[list(allowed)] = True
            assert np.array_equal(y[b][keep], x[b][keep])
            assert np.all(y[b][~keep] == neg)


def check_argmax(seed: int) -> None:
    r = np.random.default_rng(seed)
    for B, V in ((3, 1), (4, 37), (5, 1000)):
        f = r.integers(-3, 4, (B, V)).astype(np.float32)   # many exact ties
        f[0, :] = -np.inf
        got = oracle.argmax(f.view(np.uint32))
        assert got.tolist() == np.argmax(f, axis=1).tolist()   # numpy: first maximum
        bf = (f.view(np.uint32) >> 16).astype(np.uint16)        # these values are exact in bf16
        assert oracle.argmax(bf).tolist() == np.argmax(f, axis=1).tolist()


def check_golden(name: str) -> None:
    g = json.load(open(os.path.join(GOLDEN, name)))
    toks = [b"" if s == "<EOS>" else s.encode() for s in g["vocab"]]
    strings = [s.encode() for s in g["set"]]
    t, voc = build(strings, toks)
    ex = g["expect"]
    if "num_nodes" in ex:
        assert t.num_nodes == ex["num_nodes"]["value"], ex["num_nodes"]["cite"]
    if "num_chars" in ex:
        assert t.num_chars == ex["num_chars"]["value"], ex["num_chars"]["cite"]
    ids, _ = prefix_ids(strings)
    name_of = {i: g["vocab"][i] for i in range(len(toks))}
    for kind in ("rows_exact", "rows_contain"):
        for row in ex[kind]:
            n = ids[row["prefix"].encode()]
            assert t.prefix(n) == row["prefix"].encode()
            got = {name_of[v] for v in row_ids(oracle.mask_rows(t, voc, [n])[0], len(toks))}
            want = set(row["tokens"])
            if kind == "rows_exact":
                assert got == want, (row["cite"], sorted(got))
            else:
                assert want <= got, (row["cite"], sorted(got))
    # token paths from the root: every step of a path that ends on a node or
    # FINISHED is allowed by the row it leaves; the walk ends where stated
    id_of = {name: i for i, name in name_of.items()}
    ends = {"FINISHED": oracle.FINISHED, "DEAD": oracle.DEAD}
    for path in ex.get("paths", []):
        state = np.zeros(1, np.int32)
        errors = 0
        for name in path["tokens"]:
            v = id_of[name]
            if path["end"] != "DEAD" and state[0] >= 0:
                assert v in row_ids(oracle.mask_rows(t, voc, [int(state[0])])[0], len(toks)), path["cite"]
            state, e = oracle.advance(t, voc, state, np.array([v], np.int32))
            errors += e
        want = ends[path["end"]] if path["end"] in ends else ids[path["end"].encode()]
        assert int(state[0]) == want, (path["cite"], int(state[0]))
        assert errors == (1 if path["end"] == "DEAD" else 0), path["cite"]


def check_chain(s: bytes) -> None:
    """One string and the 256 single bytes: a chain, one token per row, EOS at the end."""
    toks = [bytes([b]) for b in range(256)] + [b""]
    t, voc = build([s], toks)
    m = oracle.mask_all(t, voc)
    assert t.num_nodes == len(s) + 1
    for d in range(len(s) + 1):
        got = row_ids(m[d], len(toks))
        assert got == ({s[d]} if d < len(s) else {256}), (d, got)


# ------------------------------------------------------------ fixed formats (App. K)

def fmt_case(seed: int):
    """A small format (L <= 5, each position a class of 1-3 bytes out of a
    few, 0x00 and 0xFF included) and a vocabulary over those bytes and others."""
    r = random.Random(seed)
    alpha = [0x00, 0x2D, 0x30, 0x31, 0x39, 0x61, 0xFF]
    L = r.randint(0, 5)
    cls = [sorted(r.sample(alpha, r.randint(1, 3))) for _ in range(L)]
    V = r.randint(2, 200)
    toks = []
    for _ in range(V - 1):
        n = r.choice([0, 1, 1, 2, 2, 3, 4, 6])
        pool = alpha + ([r.randrange(256)] if r.random() < 0.2 else [])
        toks.append(bytes(r.choice(pool) for _ in range(n)))
    toks.append(b"")
    return cls, toks


def fmt_bitmaps(cls: list[list[int]]) -> np.ndarray:
    out = np.zeros((len(cls), 32), np.uint8)
    for i, c in enumerate(cls):
        for b in c:
            out[i, b // 8] |= 1 << (b % 8)
    return out


def fmt_strings(cls: list[list[int]]) -> list[bytes]:
    """Every string of the format: the product of its classes."""
    import itertools
    return [bytes(t) for t in itertools.product(*cls)]


def check_fmt_masks(cls: list[list[int]], toks: list[bytes]) -> None:
    """Row p equals the prefix-set row (App. G.5 conditions) of every prefix
    of length p of the format's strings: the format's language is a finite
    set, and all its prefixes of one length share their continuations."""
    f = oracle.Format(fmt_bitmaps(cls))
    voc = oracle.Vocab(*W.pack(toks))
    V = len(toks)
    strings = fmt_strings(cls)
    ids, E = prefix_ids(strings)
    m = f.mask_all(voc)
    assert m.shape == (len(cls) + 1, (V + 31) // 32)
    for pre in ids:
        got = row_ids(m[len(pre)], V)
        assert got == expected_row(pre, toks, ids, E), (pre, sorted(got))
    m2 = f.mask_rows(voc, [oracle.FINISHED, oracle.DEAD, len(cls) + 1, -7])
    for k in range(4):
        assert row_ids(m2[k], V) == {V - 1}


def check_fmt_advance(cls: list[list[int]], toks: list[bytes], seed: int) -> None:
    """Positions move like the prefix walk: p -> len(p + bytes(v))."""
    f = oracle.Format(fmt_bitmaps(cls))
    voc = oracle.Vocab(*W.pack(toks))
    V, L = len(toks), len(cls)
    ids, E = prefix_ids(fmt_strings(cls))
    first = {}
    for pre in sorted(ids, key=lambda x: (len(x), x)):
        first.setdefault(len(pre), pre)
    r = random.Random(seed)
    B = 300
    states = np.array([r.choice([oracle.DEAD, oracle.FINISHED, L + 1, r.randint(0, L), r.randint(0, L)])
                       for _ in range(B)], np.int32)
    tokens = np.array([r.choice([-1, V, V - 1, r.randrange(V), r.randrange(V)]) for _ in range(B)], np.int32)
    got, err = f.advance(voc, states, tokens)
    inv = {i: pre for pre, i in ids.items()}
    want = []
    for s, v in zip(states.tolist(), tokens.tolist()):
        pre = first.get(s) if 0 <= s <= L else None
        nxt = expected_next(pre, ids[pre] if pre is not None else s, v, toks, ids, E)
        want.append(len(inv[nxt]) if nxt >= 0 else nxt)
    assert got.tolist() == want, [(s, v, g, w) for s, v, g, w in zip(states, tokens, got, want) if g != w][:5]
    assert err == sum(1 for s, w in zip(states, want) if w == oracle.DEAD and s != oracle.DEAD)


def check_fmt_closed_form(L: int, toks: list[bytes]) -> None:
    """Every class the full byte set: position p allows exactly the tokens of
    1..L-p bytes, and EOS at p = L."""
    f = oracle.Format(np.full((L, 32), 0xFF, np.uint8))
    voc = oracle.Vocab(*W.pack(toks))
    V = len(toks)
    m = f.mask_all(voc)
    for p in range(L + 1):
        want = {v for v in range(V - 1) if 1 <= len(toks[v]) <= L - p} | ({V - 1} if p == L else set())
        assert row_ids(m[p], V) == want, p

