"""GPU parity of the lazy rows (valid[n] computed on first visit, LRU cache;
App. H.5) through the C ABI: every row equals the oracle's, every masked
logit and state equals the dense path's, on small random cases, the K = 100
to 74,719 workloads, the 256-set forest, and with caches small enough that
rows are evicted and recomputed within one decode loop.
"""
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


@pytest.fixture(scope="session")
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_12574_gb300 import _build
    _build.build()
    T.load_library()
    oracle.build()
    return torch.device("cuda:0")


def _np_u32(t):
    import torch
    return t.cpu().contiguous().view(torch.int32).numpy().view(np.uint32)


def _bits(t):
    import torch
    t = t.cpu().contiguous()
    if t.dtype == torch.float32:
        return t.view(torch.int32).numpy().view(np.uint32)
    return t.view(torch.int16).numpy().view(np.uint16)


def _want_rows(ot, ov, states, V):
    """Oracle rows of node states; {EOS} for FINISHED, DEAD and non-node ids."""
    Wd = (V + 31) // 32
    out = np.zeros((len(states), Wd), np.uint32)
    node = (states >= 0) & (states < ot.num_nodes)
    if node.any():
        out[node] = oracle.mask_rows(ot, ov, states[node].astype(np.int32), nthreads=NCPU)
    out[~node, (V - 1) // 32] = np.uint32(1 << ((V - 1) % 32))
    return out


def _rows(cuda, h, states, V):
    import torch
    return _np_u32(T.trie_lazy_rows(h, torch.as_tensor(np.asarray(states, np.int32), device=cuda), V))


@pytest.mark.parametrize("seed", range(40))
def test_lazy_rows_small_random_exhaustive(cuda, seed):
    """Every node, plus FINISHED / DEAD / out-of-range states, twice: the
    first call computes the rows, the second takes them from the cache."""
    strings, toks = random_case(5000 + seed)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    h = T.trie_build(sb, so)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    n = ot.num_nodes
    states = np.array(list(range(n)) + [-1, -2, n, n + 3, -9, 2**31 - 1], np.int32)
    T.trie_lazy_init(h, vb, vo, V, cache_rows=4 * n + 8, max_batch=len(states))
    want = _want_rows(ot, ov, states, V)
    assert np.array_equal(_rows(cuda, h, states, V), want)
    hits, misses = T.trie_lazy_stats(h)
    assert hits == 0 and misses == n
    assert np.array_equal(_rows(cuda, h, states[::-1].copy(), V), want[::-1])
    hits, misses = T.trie_lazy_stats(h)
    # every node row of the second call is a hit, unless its set had no free
    # row in the first call (then it was computed for that call only)
    assert hits + (misses - n) == n and hits >= n // 2


@pytest.mark.parametrize("cfg", [1, 2, 3, 4])
def test_lazy_rows_config_sampled(cuda, cfg):
    """The root (whole-trie subtree), shallow nodes and random nodes."""
    w = W.config(cfg)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    ot, ov = oracle.Trie(w.set_bytes, w.set_offsets), oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    n = ot.num_nodes
    r = np.random.default_rng(cfg)
    states = np.concatenate([np.arange(min(n, 300)), r.integers(0, n, 700), [n - 1, -2, -1]]).astype(np.int32)
    T.trie_lazy_init(h, w.vocab_bytes, w.vocab_offsets, w.V, cache_rows=2048, max_batch=len(states))
    want = _want_rows(ot, ov, states, w.V)
    for _ in range(2):
        got = _rows(cuda, h, states, w.V)
        bad = np.nonzero((got != want).any(axis=1))[0]
        assert bad.size == 0, f"state {states[bad[0]]} differs"


def test_lazy_rows_long_tokens(cuda):
    """Tokens longer than 16 bytes spelled along deep paths (the path hash
    beyond the 16-label window)."""
    r = np.random.default_rng(3)
    strings = W.tool_names(3, 60, 12, lo=20, hi=48)
    toks = [bytes([b]) for b in range(256)]
    seen = set(toks)
    for _ in range(3000):
        s_ = strings[r.integers(len(strings))]
        L = int(r.integers(2, 40))
        a0 = int(r.integers(0, max(1, len(s_) - L + 1)))
        t = s_[a0:a0 + L]
        if t not in seen:
            seen.add(t)
            toks.append(t)
    toks.append(b"")
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    h = T.trie_build(sb, so)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    assert max(len(t) for t in toks) > 16 and h.max_depth > 16
    states = np.arange(ot.num_nodes, dtype=np.int32)
    T.trie_lazy_init(h, vb, vo, V, cache_rows=0, max_batch=4096)
    want = _want_rows(ot, ov, states, V)
    for a in range(0, len(states), 4096):
        assert np.array_equal(_rows(cuda, h, states[a:a + 4096], V), want[a:a + 4096])


def test_lazy_rows_forest_sampled(cuda):
    """256 per-request sets: each set's root and random nodes, rows against
    the oracle on that set's own trie."""
    w = W.config(5)
    h = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    roots = h.roots()
    T.trie_lazy_init(h, w.vocab_bytes, w.vocab_offsets, w.V, cache_rows=1024, max_batch=2048)
    rng = np.random.default_rng(5)
    sel = rng.choice(h.num_sets, 64, replace=False)
    states, want = [], []
    for i in sel:
        ot = oracle.Trie(*W.pack(strings[w.set_index[i]:w.set_index[i + 1]]))
        local = np.unique(np.concatenate([[0], rng.integers(0, ot.num_nodes, 7)])).astype(np.int32)
        want.append(oracle.mask_rows(ot, ov, local))
        states.append(local + int(roots[i]))
    states = np.concatenate(states).astype(np.int32)
    want = np.concatenate(want)
    assert np.array_equal(_rows(cuda, h, states, w.V), want)


@pytest.mark.parametrize("cfg,cache", [(1, 4096), (3, 4096), (3, 16), (3, 0), (2, 64)])
def test_lazy_decode_equals_dense(cuda, cfg, cache):
    """The workload's decode loop (greedy tokens from the dense path) through
    trie_lazy_advance_apply: logits and states bit-identical to
    trie_advance_apply's, with a cache large enough to keep every row, one
    so small that rows are evicted every step (16 rows), and none. Within one
    loop every step reaches new nodes (one level deeper), so rows are reused
    only by a second loop over the same requests."""
    import torch
    w = W.config(cfg)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    m = T.alloc_mask(h, w.V, cuda)
    T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, m)
    hl = T.trie_build(w.set_bytes, w.set_offsets)
    T.trie_lazy_init(hl, w.vocab_bytes, w.vocab_offsets, w.V, cache_rows=cache, max_batch=w.batch)
    B = w.batch
    steps = min(w.steps, 24)
    logits = [W.logits(w, s, device="cuda") for s in range(steps)]

    def one_pass():
        node_rows = 0
        st_d = torch.zeros(B, dtype=torch.int32, device=cuda)
        st_l = torch.zeros(B, dtype=torch.int32, device=cuda)
        tok = torch.zeros(B, dtype=torch.int32, device=cuda)
        err_d = torch.zeros(1, dtype=torch.int32, device=cuda)
        err_l = torch.zeros(1, dtype=torch.int32, device=cuda)
        for s in range(steps):
            xd, xl = logits[s].clone(), logits[s].clone()
            if s == 0:
                T.trie_apply_mask(h, xd, st_d)
                T.trie_lazy_apply(hl, xl, st_l)
            else:
                nd, nl = torch.empty_like(st_d), torch.empty_like(st_l)
                T.trie_advance_apply(h, st_d, tok, nd, xd, err_d)
                T.trie_lazy_advance_apply(hl, st_l, tok, nl, xl, err_l)
                st_d, st_l = nd, nl
            assert torch.equal(st_d, st_l), f"states differ at step {s}"
            node_rows += int((st_d >= 0).sum().item())
            assert np.array_equal(_bits(xd), _bits(xl)), f"masked logits differ at step {s}"
            tok = torch.argmax(xd, dim=1).to(torch.int32)
        assert int(err_d.item()) == int(err_l.item()) == 0
        return node_rows

    rows1 = one_pass()
    h1, m1 = T.trie_lazy_stats(hl)
    assert h1 + m1 == rows1
    if cache == 0:
        assert h1 == 0
    rows2 = one_pass()
    h2, m2 = T.trie_lazy_stats(hl)
    assert (h2 - h1) + (m2 - m1) == rows2
    if cache == 0:
        assert h2 == 0
    if cache >= 4096:
        assert h2 - h1 > m2 - m1     # the second loop finds most rows cached


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [33, 1001, 4096])
def test_lazy_apply_random_bits(cuda, dtype, V):
    """Allowed logits keep their exact bits (NaN payloads, -0.0); the rest
    become -inf; V = 33 and 1001 take the one-thread-per-logit path."""
    import torch
    r = np.random.default_rng(V + 7)
    strings = [bytes(r.integers(97, 100, r.integers(1, 6))) for _ in range(30)]
    toks = [bytes(r.integers(97, 100, r.integers(1, 4))) for _ in range(V - 1)] + [b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h = T.trie_build(sb, so)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    B = 37
    states = r.choice(np.array([-1, -2, ot.num_nodes, -9] + list(range(ot.num_nodes)) * 3, np.int32), B)
    if dtype == "f32":
        raw = r.integers(0, 2**32, (B, V), dtype=np.uint64).astype(np.uint32)
        x = torch.from_numpy(raw.view(np.int32)).view(torch.float32).to(cuda)
    else:
        raw = r.integers(0, 2**16, (B, V), dtype=np.uint32).astype(np.uint16)
        x = torch.from_numpy(raw.view(np.int16)).view(torch.bfloat16).to(cuda)
    want = oracle.apply(ot, ov, raw, states)
    T.trie_lazy_init(h, vb, vo, V, cache_rows=8, max_batch=B)
    T.trie_lazy_apply(h, x, torch.as_tensor(states, device=cuda))
    assert np.array_equal(_bits(x), want)


def test_lazy_lru_within_a_set(cuda):
    """cache_rows = 8 is one set: rows of the current call are never evicted,
    and a new row replaces the least recently used one."""
    strings = [bytes([97 + i]) + b"x" for i in range(20)]
    toks = [bytes([c]) for c in range(256)] + [b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    h = T.trie_build(sb, so)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    T.trie_lazy_init(h, vb, vo, V, cache_rows=8, max_batch=64)
    A = np.arange(1, 9, dtype=np.int32)      # 8 nodes: fill the set
    Bn = np.arange(9, 13, dtype=np.int32)    # 4 more: evict 4 rows of A
    for states in (A, Bn):
        assert np.array_equal(_rows(cuda, h, states, V), _want_rows(ot, ov, states, V))
    h0, m0 = T.trie_lazy_stats(h)
    assert (h0, m0) == (0, 12)
    assert np.array_equal(_rows(cuda, h, A, V), _want_rows(ot, ov, A, V))
    h1, m1 = T.trie_lazy_stats(h)
    assert (h1 - h0, m1 - m0) == (4, 4)       # 4 of A were still cached
    assert np.array_equal(_rows(cuda, h, Bn, V), _want_rows(ot, ov, Bn, V))
    # 16 distinct nodes in one call: 8 cached rows at most, the rest per-call rows
    many = np.arange(1, 17, dtype=np.int32)
    assert np.array_equal(_rows(cuda, h, np.concatenate([many, many]), V),
                          _want_rows(ot, ov, np.concatenate([many, many]), V))
    # repeated states in one call count once per batch row but compute once
    h2, m2 = T.trie_lazy_stats(h)
    assert np.array_equal(_rows(cuda, h, np.full(40, 3, np.int32), V), _want_rows(ot, ov, np.full(40, 3, np.int32), V))
    h3, m3 = T.trie_lazy_stats(h)
    assert (h3 - h2) + (m3 - m2) == 40


def test_lazy_argument_checks(cuda):
    import torch
    sb, so = W.pack([b"ab", b"b"])
    vb, vo = W.pack([b"a", b"b", b""])
    h = T.trie_build(sb, so)
    st = torch.zeros(4, dtype=torch.int32, device=cuda)
    with pytest.raises(T.TrieError) as e:
        T.trie_lazy_apply(h, torch.zeros((4, 3), device=cuda), st)
    assert e.value.code == T.TRIE_ESTATE
    T.trie_lazy_init(h, vb, vo, 3, cache_rows=8, max_batch=2)
    with pytest.raises(T.TrieError) as e:        # B > max_batch
        T.trie_lazy_apply(h, torch.zeros((4, 3), device=cuda), st)
    assert e.value.code == T.TRIE_EINVAL
    with pytest.raises(T.TrieError) as e:        # V differs
        T.trie_lazy_apply(h, torch.zeros((2, 4), device=cuda), st[:2])
    assert e.value.code == T.TRIE_EINVAL
    with pytest.raises(T.TrieError):             # states_out == states_in
        T.trie_lazy_advance_apply(h, st[:2], st[:2], st[:2], torch.zeros((2, 3), device=cuda))
    # B = 0 is a no-op; re-initialising starts with an empty cache
    T.trie_lazy_apply(h, torch.zeros((0, 3), device=cuda), st[:0])
    T.trie_lazy_init(h, vb, vo, 3, cache_rows=0, max_batch=2)
    assert T.trie_lazy_stats(h) == (0, 0)


def test_lazy_and_dense_share_the_transition_table(cuda):
    """One handle used by lazy rows and dense compiles in turn, with two
    vocabularies: lazy rows record the moves they find in the handle's
    transition table, a dense compile completes or replaces it, and every
    advance stays equal to the oracle's."""
    import torch
    w = W.config(1)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    toks_a = W.unpack(w.vocab_bytes, w.vocab_offsets)
    toks_b = toks_a[:-1][::-1] + [b""]                 # same strings, other ids
    vb_b, vo_b = W.pack(toks_b)
    ov_a = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    ov_b = oracle.Vocab(vb_b, vo_b)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    r = np.random.default_rng(11)
    B, V = 64, w.V
    n = ot.num_nodes

    def lazy_step(ov, states, tokens):
        x = torch.zeros((B, V), device=cuda)
        out = torch.empty(B, dtype=torch.int32, device=cuda)
        T.trie_lazy_advance_apply(h, torch.as_tensor(states, device=cuda), torch.as_tensor(tokens, device=cuda),
                                  out, x)
        want, _ = oracle.advance(ot, ov, states, tokens)
        assert np.array_equal(out.cpu().numpy(), want)
        return want

    def dense_step(ov, states, tokens):
        st = torch.as_tensor(states, device=cuda).clone()
        T.trie_advance(h, st, torch.as_tensor(tokens, device=cuda))
        want, _ = oracle.advance(ot, ov, states, tokens)
        assert np.array_equal(st.cpu().numpy(), want)

    def batch():
        states = r.integers(0, n, B).astype(np.int32)
        # tokens that are allowed from each state half the time
        rows = oracle.mask_rows(ot, ov_a, states)
        toks = r.integers(0, V - 1, B).astype(np.int32)
        for b in range(0, B, 2):
            ids = np.nonzero(np.unpackbits(rows[b].view(np.uint8), bitorder="little")[:V])[0]
            ids = ids[ids != V - 1]
            if ids.size:
                toks[b] = ids[r.integers(ids.size)]
        return states, toks

    T.trie_lazy_init(h, w.vocab_bytes, w.vocab_offsets, V, cache_rows=256, max_batch=B)
    for _ in range(3):                                 # the lazy rows fill the table in part
        lazy_step(ov_a, *batch())
    m = T.alloc_mask(h, V, cuda)
    T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, V, m)   # completes it
    for _ in range(2):
        dense_step(ov_a, *batch())
        lazy_step(ov_a, *batch())
    T.trie_compile_masks(h, vb_b, vo_b, V, m)          # replaces it (vocabulary b)
    s, t = batch()
    dense_step(ov_b, s, t)
    lazy_step(ov_a, s, t)                              # lazy rows keep vocabulary a, walk the bytes
    T.trie_lazy_init(h, vb_b, vo_b, V, cache_rows=256, max_batch=B)
    lazy_step(ov_b, s, t)


def test_lazy_large_batch_small_cache(cuda):
    """3,000 batch rows (more than the resolve's 1,024 threads) over a
    512-row cache, so that sets overflow into per-call rows and rows are
    evicted between calls; three calls with overlapping state sets, every
    row against the oracle."""
    w = W.config(3)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    ot, ov = oracle.Trie(w.set_bytes, w.set_offsets), oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    n = ot.num_nodes
    T.trie_lazy_init(h, w.vocab_bytes, w.vocab_offsets, w.V, cache_rows=512, max_batch=3000)
    r = np.random.default_rng(33)
    pool = r.choice(n, 1500, replace=False).astype(np.int32)
    total = 0
    for call in range(3):
        states = r.choice(pool, 3000).astype(np.int32)
        states[::97] = -2
        got = _rows(cuda, h, states, w.V)
        want = _want_rows(ot, ov, states, w.V)
        bad = np.nonzero((got != want).any(axis=1))[0]
        assert bad.size == 0, f"call {call}: state {states[bad[0]]} differs"
        total += int((states >= 0).sum())
    hits, misses = T.trie_lazy_stats(h)
    assert hits + misses == total and hits > 0
