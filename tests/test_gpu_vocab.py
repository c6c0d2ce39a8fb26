"""Vocabulary handles (trie_vocab_create / trie_compile_masks_vocab /
trie_compile_lists_vocab): the compiles that name an uploaded vocabulary give
the oracle's masks and lists, bit for bit, like the compiles that pass the
vocabulary's arrays; a handle outlives the caller's arrays and its own
release while a trie still uses it."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W
from pins import random_case

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_12574_gb300 import _build
    _build.build()
    oracle.build()
    return torch.device("cuda:0")


def _pairs(h, V):
    off, tok = T.trie_copy_lists(h)
    off = off.cpu().numpy()
    rows = np.repeat(np.arange(len(off) - 1, dtype=np.int64), np.diff(off))
    return np.sort(rows * V + tok.cpu().numpy().astype(np.int64))


def _oracle_pairs(m, V):
    rows, words = np.nonzero(m)
    out = []
    for r, w in zip(rows, words):
        x = int(m[r, w])
        while x:
            lo = x & -x
            out.append(int(r) * V + int(w) * 32 + lo.bit_length() - 1)
            x ^= lo
    return np.sort(np.array(out, np.int64))


@pytest.mark.parametrize("seed", range(6))
def test_vocab_handle_masks_and_lists_equal_oracle(cuda, seed):
    import torch
    strings, toks = random_case(7000 + seed)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    want = oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo))
    voc = T.trie_vocab_create(vb, vo, V)
    assert voc.V == V
    h = T.trie_build(sb, so)
    m = T.alloc_mask(h, V)
    T.trie_compile_masks_vocab(h, voc, m)
    got = m.cpu().numpy().view(np.uint32)
    assert np.array_equal(got, want)
    n = T.trie_compile_lists_vocab(h, voc)
    wp = _oracle_pairs(want, V)
    assert n == len(wp)
    assert np.array_equal(_pairs(h, V), wp)
    torch.cuda.synchronize()


def test_vocab_handle_offsets_not_from_zero(cuda):
    """Token bytes that start inside a larger buffer (offsets[0] > 0): the
    reversed-token trie of the list compile reads the handle's copy."""
    strings, toks = random_case(7100)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    V = len(toks)
    pad = 13
    vb2 = np.concatenate([np.full(pad, 0x7A, np.uint8), vb])
    vo2 = vo + pad
    want = oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo))
    voc = T.trie_vocab_create(vb2, vo2, V)
    h = T.trie_build(sb, so)
    n = T.trie_compile_lists_vocab(h, voc)
    wp = _oracle_pairs(want, V)
    assert n == len(wp)
    assert np.array_equal(_pairs(h, V), wp)


def test_vocab_handle_outlives_arrays_and_release(cuda):
    """The caller's arrays are overwritten after trie_vocab_create and the
    handle is released before the decode: the trie's compiled vocabulary
    stays valid for the advance (states against the oracle's)."""
    import torch
    w = W.config(1)
    vb = np.array(w.vocab_bytes, np.uint8, copy=True)
    vo = np.array(w.vocab_offsets, np.int64, copy=True)
    voc = T.trie_vocab_create(vb, vo, w.V)
    vb[:] = 0x41
    h = T.trie_build(w.set_bytes, w.set_offsets)
    m = T.alloc_mask(h, w.V)
    T.trie_compile_masks_vocab(h, voc, m)
    voc.destroy()
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    assert np.array_equal(m.cpu().numpy().view(np.uint32), oracle.mask_all(ot, ov))
    r = np.random.default_rng(5)
    states = r.integers(0, ot.num_nodes, 64).astype(np.int32)
    tokens = r.integers(0, w.V, 64).astype(np.int32)
    want, _ = oracle.advance(ot, ov, states, tokens)
    st = torch.tensor(states, device=cuda)
    T.trie_advance(h, st, torch.tensor(tokens, device=cuda))
    assert np.array_equal(st.cpu().numpy(), want)


def test_vocab_handle_fused_decode_lists(cuda):
    """The list-driven decode (apply, then fused advance + apply) after a
    compile that names a vocabulary handle: bit for bit the oracle's."""
    import torch
    w = W.config(2)
    voc = T.trie_vocab_create(w.vocab_bytes, w.vocab_offsets, w.V)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    T.trie_compile_lists_vocab(h, voc)
    logits = [W.logits(w, s, device="cuda") for s in range(w.steps)]
    bufs = [torch.zeros(w.batch, dtype=torch.int32, device=cuda) for _ in range(2)]
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    got, tok = [], None
    for t in range(w.steps):
        x = logits[t].clone()
        if t == 0:
            T.trie_apply_lists(h, x, bufs[0])
        else:
            T.trie_advance_apply_lists(h, bufs[(t - 1) % 2], tok, bufs[t % 2], x, err)
        tok = torch.argmax(x, dim=1).to(torch.int32)
        got.append((x.cpu(), tok.cpu().numpy()))
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)

    def bits(t):
        t = t.cpu().contiguous()
        return (t.view(torch.int32).numpy().view(np.uint32) if t.dtype == torch.float32
                else t.view(torch.int16).numpy().view(np.uint16))

    masked, toks, _, oerr = oracle.decode(ot, ov, (bits(lg) for lg in logits), np.zeros(w.batch, np.int32))
    for t in range(w.steps):
        assert np.array_equal(bits(got[t][0]), masked[t]), t
        assert np.array_equal(got[t][1], toks[t]), t
    assert int(err.item()) == oerr == 0
