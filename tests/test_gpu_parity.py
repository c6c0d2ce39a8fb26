"""GPU parity: libtriemask (through its C ABI) against the CPU oracle, bit for bit.

Masks, states and masked logits must be identical to the oracle's on the same
seeded inputs: small random sets (exhaustive), the K=100 / 1,000 / 10,000 /
74,719 workloads in full, and the 256-request forest on sampled rows.
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
    """Raw bits of a CPU/GPU float tensor as a numpy array (uint32 or uint16)."""
    import torch
    t = t.cpu().contiguous()
    if t.dtype == torch.float32:
        return t.view(torch.int32).numpy().view(np.uint32)
    return t.view(torch.int16).numpy().view(np.uint16)


def _compile(cuda, set_bytes, set_offsets, vocab_bytes, vocab_offsets, forest_index=None):
    V = len(vocab_offsets) - 1
    if forest_index is None:
        h = T.trie_build(set_bytes, set_offsets)
    else:
        h = T.trie_build_many(set_bytes, set_offsets, forest_index)
    m = T.alloc_mask(h, V, cuda)
    T.trie_compile_masks(h, vocab_bytes, vocab_offsets, V, m)
    return h, m


def _first_diff(a, b):
    rows = np.nonzero((a != b).any(axis=1))[0]
    return None if rows.size == 0 else int(rows[0])


@pytest.mark.parametrize("seed", range(60))
def test_compile_small_random_exhaustive(cuda, seed):
    strings, toks = random_case(1000 + seed)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h, m = _compile(cuda, sb, so, vb, vo)
    want = oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo))
    got = _np_u32(m)
    assert got.shape == want.shape
    assert _first_diff(got, want) is None, _first_diff(got, want)


@pytest.mark.parametrize("seed", range(30))
def test_compile_small_random_unique_tokens(cuda, seed):
    """Vocabularies without repeated token strings: the per-node search then
    accepts a key found in its first slot pair without probing further."""
    strings, toks = random_case(3000 + seed)
    uniq = list(dict.fromkeys(t for t in toks[:-1] if t)) + [b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(uniq)
    h, m = _compile(cuda, sb, so, vb, vo)
    want = oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo))
    assert _first_diff(_np_u32(m), want) is None


def test_compile_repeated_tokens_large_vocab(cuda):
    """The K=100 workload's vocabulary with 2,000 of its tokens repeated at
    the end: every copy of an allowed token must be allowed too."""
    w = W.config(1)
    r = np.random.default_rng(7)
    toks = [bytes(w.vocab_bytes[w.vocab_offsets[i]:w.vocab_offsets[i + 1]]) for i in range(w.V - 1)]
    toks += [toks[int(i)] for i in r.integers(0, len(toks), 2000)] + [b""]
    vb, vo = W.pack(toks)
    h, m = _compile(cuda, w.set_bytes, w.set_offsets, vb, vo)
    want = oracle.mask_all(oracle.Trie(w.set_bytes, w.set_offsets), oracle.Vocab(vb, vo), nthreads=NCPU)
    assert _first_diff(_np_u32(m), want) is None


@pytest.mark.parametrize("cfg", [1, 2, 3, 4])
def test_compile_config_full(cuda, cfg):
    """Every row of the full-size workloads, compared in row blocks."""
    w = W.config(cfg)
    h, m = _compile(cuda, w.set_bytes, w.set_offsets, w.vocab_bytes, w.vocab_offsets)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    assert h.num_nodes == ot.num_nodes
    step = 4096
    for r0 in range(0, h.num_nodes, step):
        rows = np.arange(r0, min(r0 + step, h.num_nodes), dtype=np.int32)
        want = oracle.mask_rows(ot, ov, rows, nthreads=NCPU)
        got = _np_u32(m[r0:r0 + len(rows)])
        d = _first_diff(got, want)
        assert d is None, f"row {r0 + d} differs"


@pytest.mark.parametrize("seed", range(4))
def test_compile_long_suffixes(cuda, seed):
    """Deep paths and tokens longer than 16 bytes (the search beyond the
    16-label window), both compile entry points."""
    import torch
    r = np.random.default_rng(seed)
    strings = W.tool_names(seed, 60, 12, lo=20, hi=48)
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
    h, m = _compile(cuda, sb, so, vb, vo)
    want = oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo), nthreads=NCPU)
    assert max(len(t) for t in toks) > 16 and h.max_depth > 16
    assert _first_diff(_np_u32(m), want) is None
    m2 = torch.full_like(m, -1)
    T.trie_compile_masks_noalloc(h, vb, vo, V, m2)
    assert _first_diff(_np_u32(m2), want) is None


def test_compile_many_hits_per_node(cuda):
    """a^k for k = 1..24 are all tokens: deep nodes of a run of 'a's end more
    than 16 allowed (row, token) pairs (the hit buffer's overflow path)."""
    strings = [b"a" * 30, b"a" * 12 + b"b", b"ab" * 10]
    toks = [bytes([b]) for b in range(256)] + [b"a" * k for k in range(2, 25)] + [b"ab", b"aab", b"ba" * 3, b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h, m = _compile(cuda, sb, so, vb, vo)
    want = oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo))
    assert _first_diff(_np_u32(m), want) is None


def test_compile_forest_sampled(cuda):
    """256 per-request sets (4.8M nodes, 76 GB mask): sampled rows of every set."""
    import torch
    w = W.config(5)
    h, m = _compile(cuda, w.set_bytes, w.set_offsets, w.vocab_bytes, w.vocab_offsets, w.set_index)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    rng = np.random.default_rng(5)
    roots = h.roots()
    for i in range(h.num_sets):
        st = strings[w.set_index[i]:w.set_index[i + 1]]
        ot = oracle.Trie(*W.pack(st))
        n = ot.num_nodes
        local = np.unique(np.concatenate([[0, n - 1], rng.integers(0, n, 6)])).astype(np.int32)
        want = oracle.mask_rows(ot, ov, local)
        idx = torch.as_tensor(local.astype(np.int64) + int(roots[i]), device=cuda)
        got = _np_u32(m.index_select(0, idx))
        assert _first_diff(got, want) is None, f"set {i}"
    del m
    torch.cuda.empty_cache()


def _gpu_decode(cuda, h, logits, states0):
    import torch
    st = torch.as_tensor(states0, dtype=torch.int32, device=cuda).clone()
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    out = []
    for lg in logits:
        x = lg.clone()
        T.trie_apply_mask(h, x, st)
        tok = torch.argmax(x, dim=1).to(torch.int32)
        T.trie_advance(h, st, tok, err)
        out.append((x, tok.cpu().numpy(), st.cpu().numpy().copy()))
    return out, int(err.item())


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_decode_loop_config(cuda, cfg):
    """apply -> greedy argmax -> advance for every step of the workload, bit for bit."""
    w = W.config(cfg)
    h, m = _compile(cuda, w.set_bytes, w.set_offsets, w.vocab_bytes, w.vocab_offsets)
    logits = [W.logits(w, s, device="cuda") for s in range(w.steps)]
    states0 = np.zeros(w.batch, np.int32)
    got, gerr = _gpu_decode(cuda, h, logits, states0)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    masked, toks, sts, oerr = oracle.decode(ot, ov, (_bits(lg) for lg in logits), states0)
    for s in range(w.steps):
        assert np.array_equal(_bits(got[s][0]), masked[s]), f"masked logits differ at step {s}"
        assert np.array_equal(got[s][1], toks[s]), f"tokens differ at step {s}"
        assert np.array_equal(got[s][2], sts[s]), f"states differ at step {s}"
    assert gerr == oerr == 0
    # 100% validity: every request that finished emitted a set member
    strings = set(W.unpack(w.set_bytes, w.set_offsets))
    tokb = W.unpack(w.vocab_bytes, w.vocab_offsets)
    for b in range(w.batch):
        if sts[-1][b] == oracle.FINISHED:
            out = b"".join(tokb[toks[s][b]] for s in range(w.steps) if toks[s][b] != w.V - 1)
            assert out in strings


@pytest.mark.parametrize("seed", range(20))
def test_advance_random(cuda, seed):
    import torch
    strings, toks = random_case(2000 + seed)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    h, m = _compile(cuda, sb, so, vb, vo)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    r = np.random.default_rng(seed)
    B = 1000
    n = ot.num_nodes
    states = r.choice(np.array([-1, -2, n, n + 5, -7] + list(range(n)) * 4, np.int32), B)
    tokens = r.choice(np.array([-1, V, V - 1] + list(range(V)) * 3, np.int32), B)
    want, werr = oracle.advance(ot, ov, states, tokens)
    ds = torch.as_tensor(states, device=cuda).clone()
    dt = torch.as_tensor(tokens, device=cuda)
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    T.trie_advance(h, ds, dt, err)
    assert np.array_equal(ds.cpu().numpy(), want)
    assert int(err.item()) == werr


def test_advance_long_paths(cuda):
    """Tokens that walk many edges (the whole string at once)."""
    import torch
    w = W.config(2)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    toks = [bytes([b]) for b in range(256)] + strings[:200] + [b""]
    vb, vo = W.pack(toks)
    h, m = _compile(cuda, w.set_bytes, w.set_offsets, vb, vo)
    ot, ov = oracle.Trie(w.set_bytes, w.set_offsets), oracle.Vocab(vb, vo)
    states = np.zeros(200, np.int32)
    tokens = np.arange(256, 456, dtype=np.int32)
    want, _ = oracle.advance(ot, ov, states, tokens)
    ds = torch.as_tensor(states, device=cuda).clone()
    T.trie_advance(h, ds, torch.as_tensor(tokens, device=cuda))
    assert np.array_equal(ds.cpu().numpy(), want)
    assert all(ot.terminal[s] for s in want)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [2, 33, 1001, 4096, 32000])
def test_apply_random_bits(cuda, dtype, V):
    """Every bit pattern (NaN payloads, -0.0) of an allowed logit survives; the rest become -inf.
    V = 33 and 1001 take the unaligned one-thread-per-logit path."""
    import torch
    r = np.random.default_rng(V)
    strings = [bytes(r.integers(97, 100, r.integers(1, 6))) for _ in range(30)]
    toks = [bytes(r.integers(97, 100, r.integers(1, 4))) for _ in range(V - 1)] + [b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h, m = _compile(cuda, sb, so, vb, vo)
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
    T.trie_apply_mask(h, x, torch.as_tensor(states, device=cuda))
    assert np.array_equal(_bits(x), want)


def test_apply_unaligned_base_uses_scalar_path(cuda):
    import torch
    sb, so = W.pack([b"ab", b"b"])
    toks = [bytes([c]) for c in range(256)] + [b"ab"] * 7 + [b""]
    vb, vo = W.pack(toks)
    V = len(toks)
    assert V % 8 == 0
    h, m = _compile(cuda, sb, so, vb, vo)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    buf = torch.randn(3 * V + 1, device=cuda).to(torch.bfloat16)
    x = buf[1:].view(3, V)                     # 2-byte aligned rows
    st = np.array([0, 1, -2], np.int32)
    want = oracle.apply(ot, ov, _bits(x), st)
    T.trie_apply_mask(h, x, torch.as_tensor(st, device=cuda))
    assert np.array_equal(_bits(x), want)


def test_edge_cases(cuda):
    import torch
    toks = [b"a", b"b", b"ab", b""]
    vb, vo = W.pack(toks)
    # empty set: a lone, non-terminal root allows nothing
    h, m = _compile(cuda, *W.pack([]), vb, vo)
    assert h.num_nodes == 1 and _np_u32(m).tolist() == [[0]]
    # {""}: root terminal, EOS only
    h, m = _compile(cuda, *W.pack([b""]), vb, vo)
    assert _np_u32(m).tolist() == [[1 << 3]]
    # V = 2: one token plus EOS
    vb2, vo2 = W.pack([b"a", b""])
    h, m = _compile(cuda, *W.pack([b"a", b""]), vb2, vo2)
    assert _np_u32(m).tolist() == [[0b11], [0b10]]
    # B = 0 is a no-op
    e = torch.empty(0, dtype=torch.int32, device=cuda)
    T.trie_advance(h, e, e)
    T.trie_apply_mask(h, torch.empty((0, 2), device=cuda), e)
    # V mismatch and unknown dtype are rejected
    with pytest.raises(T.TrieError):
        T.trie_apply_mask(h, torch.zeros((1, 3), device=cuda), torch.zeros(1, dtype=torch.int32, device=cuda))


def test_recompile_other_vocab_same_handle(cuda):
    """A handle compiled twice uses the latest vocabulary and mask; cached
    vocabularies are reused only for identical arrays."""
    w = W.config(1)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    for seed in (0, 7, 0):
        spec = W.VocabSpec(V=5000, max_len=12, substr_frac=0.3, run_frac=0.0, run_len=(2, 4),
                           upper=False, mixed=False)
        vb, vo = W.byte_vocab(seed, spec, substr_src=W.tool_stems(0, 40))
        m = T.alloc_mask(h, 5000, cuda)
        T.trie_compile_masks(h, vb, vo, 5000, m)
        want = oracle.mask_all(ot, oracle.Vocab(vb, vo), nthreads=NCPU)
        assert np.array_equal(_np_u32(m), want)


def test_mask_offset_pointer(cuda):
    """A mask that starts 4 bytes past a 16-byte boundary (scalar head words)."""
    import torch
    w = W.config(1)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    Wd = T.mask_words(w.V)
    buf = torch.zeros(h.num_nodes * Wd + 4, dtype=torch.int32, device=cuda)
    m = buf[1:1 + h.num_nodes * Wd].view(h.num_nodes, Wd)
    T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, m)
    want = oracle.mask_all(oracle.Trie(w.set_bytes, w.set_offsets),
                           oracle.Vocab(w.vocab_bytes, w.vocab_offsets), nthreads=NCPU)
    assert np.array_equal(_np_u32(m), want)
    assert int(buf[0].item()) == 0 and int(buf[-3:].abs().sum().item()) == 0


def test_compile_forest_full(cuda):
    """256 per-request sets (4.8M nodes, 76 GB mask): every row of every set,
    against the oracle's pairs (each set's Aho-Corasick pairs plus EOS at its
    terminal nodes, offset by its root), compared on the device in chunks."""
    import torch
    from maskcheck import assert_mask_equals_pairs, forest_pairs
    w = W.config(5)
    h, m = _compile(cuda, w.set_bytes, w.set_offsets, w.vocab_bytes, w.vocab_offsets, w.set_index)
    ac = oracle.AhoCorasick(oracle.Vocab(w.vocab_bytes, w.vocab_offsets))
    rows, toks = forest_pairs(ac, W.unpack(w.set_bytes, w.set_offsets), w.set_index, h.roots(), w.V,
                              nthreads=NCPU)
    torch.cuda.synchronize()
    assert_mask_equals_pairs(m, rows, toks)
    del m
    torch.cuda.empty_cache()


def test_decode_loop_forest(cuda):
    """The 256-request workload decoded as the bench decodes it: one forest of
    the requests' sets, valid lists, the list-driven apply for step 0 and one
    advance + apply launch per later step, greedy argmax in between. Every
    request is then decoded by the oracle on its own set's trie (local node id
    = forest id - the set's root) and compared at each of the 32 steps:
    masked logits, token and state, and the error count."""
    import torch
    from concurrent.futures import ThreadPoolExecutor
    w = W.config(5)
    B, S = w.batch, w.steps
    h = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index)
    assert h.num_sets == B
    T.trie_compile_lists(h, w.vocab_bytes, w.vocab_offsets, w.V)
    roots = h.roots().astype(np.int64)
    bufs = [torch.as_tensor(roots.astype(np.int32), device=cuda), torch.empty(B, dtype=torch.int32, device=cuda)]
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    raw, masked, toks, entering = [], [], [], []
    tok = None
    for t in range(S):
        x = W.logits(w, t, device="cuda")
        raw.append(_bits(x).copy())
        if t == 0:
            T.trie_apply_lists(h, x, bufs[0])
        else:
            T.trie_advance_apply_lists(h, bufs[(t - 1) % 2], tok, bufs[t % 2], x, err)
        tok = torch.argmax(x, dim=1).to(torch.int32)
        masked.append(_bits(x).copy())
        toks.append(tok.cpu().numpy().copy())
        entering.append(bufs[t % 2].cpu().numpy().copy())
    T.trie_advance(h, bufs[(S - 1) % 2], tok, err)
    entering.append(bufs[(S - 1) % 2].cpu().numpy().copy())     # the states after the last step
    gpu_err = int(err.item())

    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    strings = W.unpack(w.set_bytes, w.set_offsets)

    def check(b):
        ot = oracle.Trie(*W.pack(strings[w.set_index[b]:w.set_index[b + 1]]))
        om, otk, ost, oe = oracle.decode(ot, ov, [raw[t][b:b + 1] for t in range(S)], np.zeros(1, np.int32))
        for t in range(S):
            g = int(entering[t + 1][b])
            g = g - int(roots[b]) if g >= 0 else g
            if not np.array_equal(masked[t][b], om[t][0]):
                return f"request {b}, step {t}: masked logits"
            if int(toks[t][b]) != int(otk[t][0]):
                return f"request {b}, step {t}: token"
            if g != int(ost[t][0]):
                return f"request {b}, step {t}: state {g} against {int(ost[t][0])}"
        return oe

    with ThreadPoolExecutor(max_workers=NCPU) as ex:
        res = list(ex.map(check, range(B)))
    bad = [r for r in res if isinstance(r, str)]
    assert not bad, bad[:5]
    assert gpu_err == sum(res) == 0
    assert int(entering[0].astype(np.int64).sum()) == int(roots.sum())   # every request starts at its root


@pytest.mark.parametrize("name", ["appG1_worked_example.json", "fig2_alignment.json",
                                  "appH9_noncanonical.json", "sec42_prefix_values.json"])
def test_golden_examples(cuda, name):
    """The paper's worked examples (tests/golden): the GPU mask equals the
    oracle's, and the GPU walks every listed token path to the oracle's state."""
    import json
    import torch
    g = json.load(open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", name)))
    toks = [b"" if s == "<EOS>" else s.encode() for s in g["vocab"]]
    sb, so = W.pack([s.encode() for s in g["set"]])
    vb, vo = W.pack(toks)
    h, m = _compile(cuda, sb, so, vb, vo)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    assert np.array_equal(_np_u32(m), oracle.mask_all(ot, ov))
    id_of = {s: i for i, s in enumerate(g["vocab"])}
    for path in g["expect"].get("paths", []):
        st = torch.zeros(1, dtype=torch.int32, device=cuda)
        err = torch.zeros(1, dtype=torch.int32, device=cuda)
        want = np.zeros(1, np.int32)
        for s in path["tokens"]:
            tok = np.array([id_of[s]], np.int32)
            T.trie_advance(h, st, torch.as_tensor(tok, device=cuda), err)
            want, _ = oracle.advance(ot, ov, want, tok)
        assert int(st.item()) == int(want[0]), path["cite"]
        assert int(err.item()) == (1 if path["end"] == "DEAD" else 0), path["cite"]
