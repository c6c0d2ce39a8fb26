"""GPU parity of the pairwise compile (trie_compile_masks_pairwise: one walk
per (node, token) pair, a warp ballot per mask word) against the CPU oracle,
bit for bit: small random sets exhaustively, deep tries with long tokens, and
the K=100 / 1,000 / 10,000 workloads in full."""
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


def _np_u32(t):
    import torch
    return t.cpu().contiguous().view(torch.int32).numpy().view(np.uint32)


def _pairwise(cuda, sb, so, vb, vo):
    import torch
    V = len(vo) - 1
    h = T.trie_build(sb, so)
    m = torch.full((h.num_nodes, T.mask_words(V)), -1, dtype=torch.int32, device=cuda)
    T.trie_compile_masks_pairwise(h, vb, vo, V, m)
    return h, _np_u32(m)


@pytest.mark.parametrize("seed", range(20))
def test_pairwise_small_random(cuda, seed):
    strings, toks = random_case(5000 + seed)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    _, got = _pairwise(cuda, sb, so, vb, vo)
    want = oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo))
    assert np.array_equal(got, want)


def test_pairwise_long_tokens(cuda):
    """Tokens of up to 40 bytes (walks past the first 16 bytes) in a deep trie."""
    r = np.random.default_rng(3)
    alpha = np.frombuffer(b"abc", np.uint8)
    strings = [bytes(r.choice(alpha, r.integers(1, 60))) for _ in range(30)]
    toks = [bytes([c]) for c in range(256)] + [s_[i:i + L] for s_ in strings for i in (0, 3)
                                               for L in (18, 25, 40) if len(s_) >= i + L] + [b""]
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    _, got = _pairwise(cuda, sb, so, vb, vo)
    assert np.array_equal(got, oracle.mask_all(oracle.Trie(sb, so), oracle.Vocab(vb, vo)))


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_pairwise_configs(cuda, cfg):
    w = W.config(cfg)
    h, got = _pairwise(cuda, w.set_bytes, w.set_offsets, w.vocab_bytes, w.vocab_offsets)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    step = 4096
    for r0 in range(0, h.num_nodes, step):
        rows = np.arange(r0, min(r0 + step, h.num_nodes), dtype=np.int32)
        assert np.array_equal(got[r0:r0 + len(rows)], oracle.mask_rows(ot, ov, rows, nthreads=NCPU)), r0
