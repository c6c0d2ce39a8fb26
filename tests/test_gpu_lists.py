"""GPU parity of the sparse valid lists (trie_compile_lists / trie_apply_lists)
against the CPU oracle: the (node, token) entries equal the oracle's, and the
list-driven mask application and decode loop are bit-identical to the
oracle's."""
from __future__ import annotations

import os

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W
from pins import random_case

pytestmark = pytest.mark.gpu
NCPU = os.cpu_count() or 1


@pytest.fixture(scope="module")
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_12574_gb300 import _build
    _build.build()
    oracle.build()
    return torch.device("cuda:0")


def _bits(t):
    import torch
    t = t.cpu().contiguous()
    if t.dtype == torch.float32:
        return t.view(torch.int32).numpy().view(np.uint32)
    return t.view(torch.int16).numpy().view(np.uint16)


def _gpu_pairs(h):
    off, tok = T.trie_copy_lists(h)
    off = off.cpu().numpy()
    tok = tok.cpu().numpy()
    rows = np.repeat(np.arange(len(off) - 1, dtype=np.int64), np.diff(off))
    assert len(rows) == len(tok) == T.trie_num_valid(h)
    return rows, tok.astype(np.int64)


def _key(rows, toks, V):
    return np.sort(rows.astype(np.int64) * V + toks.astype(np.int64))


def _oracle_pairs_from_mask(m, V):
    r, w, b = [], [], []
    rows, words = np.nonzero(m)
    for rr, ww in zip(rows, words):
        x = int(m[rr, ww])
        while x:
            lo = x & -x
            r.append(rr)
            w.append(ww * 32 + lo.bit_length() - 1)
            x ^= lo
    return np.array(r, np.int64), np.array(w, np.int64)


@pytest.mark.parametrize("seed", range(30))
def test_lists_small_random(cuda, seed):
    strings, toks = random_case(1000 + seed)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    h = T.trie_build(sb, so)
    n = T.trie_compile_lists(h, vb, vo, V)
    want = _oracle_pairs_from_mask(oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo)), V)
    got = _gpu_pairs(h)
    assert n == len(want[0])
    assert np.array_equal(_key(*got, V), _key(*want, V))


@pytest.mark.parametrize("cfg", [1, 2, 3, 4])
def test_lists_configs(cuda, cfg):
    """Every entry of the full-size workloads against the paper-algorithm pairs
    (oracle/ac.c, itself equal to the brute-force oracle) plus EOS at terminals."""
    w = W.config(cfg)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    T.trie_compile_lists(h, w.vocab_bytes, w.vocab_offsets, w.V)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    rows, toks = oracle.AhoCorasick(oracle.Vocab(w.vocab_bytes, w.vocab_offsets)).pairs(ot, nthreads=NCPU)
    term = np.nonzero(ot.terminal)[0]
    want_r = np.concatenate([rows, term]).astype(np.int64)
    want_t = np.concatenate([toks, np.full(len(term), w.V - 1)]).astype(np.int64)
    got = _gpu_pairs(h)
    assert np.array_equal(_key(*got, w.V), _key(want_r, want_t, w.V))


@pytest.mark.parametrize("seed", range(3))
def test_lists_long_tokens_deep_trie(cuda, seed):
    """Tokens longer than 16 bytes in a trie deeper than 16: the walk leaves
    the 16-label window and climbs parent links; repeated token strings are
    listed under every id."""
    r = np.random.default_rng(77 + seed)
    alpha = np.frombuffer(b"ab", np.uint8)
    strings = [bytes(r.choice(alpha, r.integers(1, 48))) for _ in range(40)]
    toks = [bytes([c]) for c in range(256)]
    toks += [bytes(r.choice(alpha, r.integers(2, 31))) for _ in range(400)]
    toks += [s_[i:i + L] for s_ in strings[:10] for i in range(0, 5) for L in (17, 23, 30) if len(s_) >= i + L]
    toks += toks[300:320]  # repeated strings
    toks.append(b"")
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    h = T.trie_build(sb, so)
    n = T.trie_compile_lists(h, vb, vo, V)
    want = _oracle_pairs_from_mask(oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo)), V)
    assert n == len(want[0])
    assert np.array_equal(_key(*_gpu_pairs(h), V), _key(*want, V))


def test_lists_many_repeated_tokens(cuda):
    """One token string under 20,000 ids: the bound on the entries (one per
    id and length) is too large to allocate, so the list compile reads the
    exact count back between its two walks."""
    r = np.random.default_rng(5)
    alpha = np.frombuffer(b"ab", np.uint8)
    strings = [bytes(r.choice(alpha, r.integers(10, 30))) for _ in range(100)]
    toks = [bytes([c]) for c in range(256)] + [b"ab"] * 20000 + [b"ba", b"aab", b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    h = T.trie_build(sb, so)
    assert h.num_nodes * (16 * 20000 + 1) > (1 << 28)
    n = T.trie_compile_lists(h, vb, vo, V)
    want = _oracle_pairs_from_mask(oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo)), V)
    assert n == len(want[0])
    assert np.array_equal(_key(*_gpu_pairs(h), V), _key(*want, V))


def test_lists_forest(cuda):
    """The 256-request forest: every set's entries, offset by its root."""
    w = W.config(5)
    h = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index)
    T.trie_compile_lists(h, w.vocab_bytes, w.vocab_offsets, w.V)
    got_r, got_t = _gpu_pairs(h)
    got = _key(got_r, got_t, w.V)
    ac = oracle.AhoCorasick(oracle.Vocab(w.vocab_bytes, w.vocab_offsets))
    strings = W.unpack(w.set_bytes, w.set_offsets)
    roots = h.roots()
    parts_r, parts_t = [], []
    for i in range(h.num_sets):
        ot = oracle.Trie(*W.pack(strings[w.set_index[i]:w.set_index[i + 1]]))
        r, t = ac.pairs(ot, nthreads=NCPU)
        term = np.nonzero(ot.terminal)[0]
        parts_r += [r.astype(np.int64) + roots[i], term.astype(np.int64) + roots[i]]
        parts_t += [t.astype(np.int64), np.full(len(term), w.V - 1, np.int64)]
    want = _key(np.concatenate(parts_r), np.concatenate(parts_t), w.V)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [2, 33, 1001, 8193, 32000])
def test_apply_lists_random_bits(cuda, dtype, V):
    import torch
    r = np.random.default_rng(V + 7)
    strings = [bytes(r.integers(97, 100, r.integers(1, 6))) for _ in range(30)]
    toks = [bytes(r.integers(97, 100, r.integers(1, 4))) for _ in range(V - 1)] + [b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h = T.trie_build(sb, so)
    T.trie_compile_lists(h, vb, vo, V)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    B = 19
    states = r.choice(np.array([-1, -2, ot.num_nodes, -9] + list(range(ot.num_nodes)) * 3, np.int32), B)
    if dtype == "f32":
        raw = r.integers(0, 2**32, (B, V), dtype=np.uint64).astype(np.uint32)
        x = torch.from_numpy(raw.view(np.int32)).view(torch.float32).to(cuda)
    else:
        raw = r.integers(0, 2**16, (B, V), dtype=np.uint32).astype(np.uint16)
        x = torch.from_numpy(raw.view(np.int16)).view(torch.bfloat16).to(cuda)
    want = oracle.apply(ot, ov, raw, states)
    T.trie_apply_lists(h, x, torch.as_tensor(states, device=cuda))
    assert np.array_equal(_bits(x), want)


@pytest.mark.parametrize("cfg", [1, 3])
def test_decode_loop_lists(cuda, cfg):
    """apply (from lists) -> greedy argmax -> advance, bit for bit at every step."""
    import torch
    w = W.config(cfg)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    T.trie_compile_lists(h, w.vocab_bytes, w.vocab_offsets, w.V)
    logits = [W.logits(w, s, device="cuda") for s in range(w.steps)]
    st = torch.zeros(w.batch, dtype=torch.int32, device=cuda)
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    got = []
    for lg in logits:
        x = lg.clone()
        T.trie_apply_lists(h, x, st)
        tok = torch.argmax(x, dim=1).to(torch.int32)
        T.trie_advance(h, st, tok, err)
        got.append((x, tok.cpu().numpy(), st.cpu().numpy().copy()))
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    masked, toks, sts, oerr = oracle.decode(ot, ov, (_bits(lg) for lg in logits), np.zeros(w.batch, np.int32))
    for s in range(w.steps):
        assert np.array_equal(_bits(got[s][0]), masked[s]), s
        assert np.array_equal(got[s][1], toks[s]), s
        assert np.array_equal(got[s][2], sts[s]), s
    assert int(err.item()) == oerr == 0


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_decode_loop_lists_fused(cuda, cfg):
    """trie_apply_lists for step 0, then trie_advance_apply_lists for every
    later step (one launch each), greedy argmax in between: masked logits,
    tokens and states bit for bit equal to the oracle's at every step."""
    import torch
    w = W.config(cfg)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    T.trie_compile_lists(h, w.vocab_bytes, w.vocab_offsets, w.V)
    logits = [W.logits(w, s, device="cuda") for s in range(w.steps)]
    bufs = [torch.zeros(w.batch, dtype=torch.int32, device=cuda) for _ in range(2)]
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    got = []
    tok = None
    for t in range(w.steps):
        x = logits[t].clone()
        if t == 0:
            T.trie_apply_lists(h, x, bufs[0])
        else:
            T.trie_advance_apply_lists(h, bufs[(t - 1) % 2], tok, bufs[t % 2], x, err)
        tok = torch.argmax(x, dim=1).to(torch.int32)
        got.append((x, tok.cpu().numpy(), bufs[t % 2].cpu().numpy().copy()))
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    masked, toks, sts, oerr = oracle.decode(ot, ov, (_bits(lg) for lg in logits), np.zeros(w.batch, np.int32))
    for t in range(w.steps):
        assert np.array_equal(_bits(got[t][0]), masked[t]), t
        assert np.array_equal(got[t][1], toks[t]), t
        if t > 0:
            assert np.array_equal(got[t][2], sts[t - 1]), t
    assert int(err.item()) == oerr == 0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [33, 1001, 8193])
def test_advance_apply_lists_random(cuda, dtype, V):
    """Random states (invalid ones included) and tokens, the scalar path for
    V = 33 / 1001: states against the oracle's advance, logits against its
    apply by the new states."""
    import torch
    r = np.random.default_rng(V + 3)
    strings = [bytes(r.integers(97, 100, r.integers(1, 6))) for _ in range(40)]
    toks = [bytes(r.integers(97, 100, r.integers(1, 4))) for _ in range(V - 1)] + [b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h = T.trie_build(sb, so)
    T.trie_compile_lists(h, vb, vo, V)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    B = 41
    states = r.choice(np.array([-1, -2, ot.num_nodes, -9] + list(range(ot.num_nodes)) * 3, np.int32), B)
    tokens = r.choice(np.array([-1, V, V - 1] + list(range(V)) * 2, np.int32), B)
    want_st, want_err = oracle.advance(ot, ov, states, tokens)
    if dtype == "f32":
        raw = r.integers(0, 2**32, (B, V), dtype=np.uint64).astype(np.uint32)
        x = torch.from_numpy(raw.view(np.int32)).view(torch.float32).to(cuda)
    else:
        raw = r.integers(0, 2**16, (B, V), dtype=np.uint32).astype(np.uint16)
        x = torch.from_numpy(raw.view(np.int16)).view(torch.bfloat16).to(cuda)
    out = torch.empty(B, dtype=torch.int32, device=cuda)
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    T.trie_advance_apply_lists(h, torch.as_tensor(states, device=cuda), torch.as_tensor(tokens, device=cuda), out, x,
                               err)
    assert np.array_equal(out.cpu().numpy(), want_st)
    assert int(err.item()) == want_err
    assert np.array_equal(_bits(x), oracle.apply(ot, ov, raw, want_st))


def test_lists_errors(cuda):
    import torch
    sb, so = W.pack([b"ab"])
    h = T.trie_build(sb, so)
    assert T.trie_num_valid(h) == -1
    with pytest.raises(T.TrieError):
        T.trie_apply_lists(h, torch.zeros((1, 4), device=cuda), torch.zeros(1, dtype=torch.int32, device=cuda))
    vb, vo = W.pack([b"a", b"b", b"ab", b""])
    assert T.trie_compile_lists(h, vb, vo, 4) == 4   # root: a, ab; 'a': b; 'ab': EOS
    with pytest.raises(T.TrieError):
        T.trie_apply_lists(h, torch.zeros((1, 5), device=cuda), torch.zeros(1, dtype=torch.int32, device=cuda))
