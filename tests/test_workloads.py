"""The seeded synthetic workloads match the recipe they are documented with.

Five workloads stand in for the paper's tool-name sets, ICD-style code lists,
tokenizers and per-query sets; each is checked here against its stated
shape: sizes, alphabets, length ranges, the code pattern, the token layout
(the 256 single bytes first, distinct multi-byte tokens, a byte-less EOS at
V - 1), the decode batch / steps / dtype / logit scale, and the node counts
the measurements quote. The generators hold no part of the method.
"""
from __future__ import annotations

import re

import numpy as np
import pytest

from paper_2608_12574_gb300 import workloads as W

CODES3 = re.compile(rb"[A-Z][0-9]{2}(\.[A-Z0-9]{1,4})?")
CODES4 = re.compile(rb"[A-Z][0-9]{2}(\.[A-Z0-9]{1,3})?")
SNAKE = re.compile(rb"[a-z_]+")


@pytest.fixture(scope="module", params=[1, 2, 3, 4, 5])
def wl(request):
    w = W.config(request.param)
    return request.param, w, W.unpack(w.set_bytes, w.set_offsets), W.unpack(w.vocab_bytes, w.vocab_offsets)


SHAPE = {  # K (strings), V, batch, steps, dtype, logit std, token lengths, name
    1: (100, 32000, 1, 64, "f32", 1.0, (2, 12), "tools-K100-V32000-B1-f32"),
    2: (1000, 128000, 64, 128, "bf16", 2.0, (2, 16), "tools-K1000-V128000-B64-bf16"),
    3: (10000, 152064, 256, 16, "bf16", 2.0, (2, 16), "icd-K10000-V152064-B256-bf16"),
    4: (74719, 262144, 256, 16, "f32", 1.0, (2, 24), "icd-K74719-V262144-B256-f32"),
    5: (None, 128000, 256, 32, "bf16", 2.0, (2, 16), "dynamic-256x(K300-2000)-V128000-B256-bf16"),
}


def test_decode_shape(wl):
    cfg, w, strings, toks = wl
    K, V, B, S, dt, std, _, name = SHAPE[cfg]
    assert w.name == name and (w.V, w.batch, w.steps, w.dtype, w.logit_std) == (V, B, S, dt, std)
    if K is not None:
        assert w.K == K


def test_vocabulary_layout(wl):
    cfg, w, _, toks = wl
    lo, hi = SHAPE[cfg][6]
    assert len(toks) == w.V
    assert all(toks[b] == bytes([b]) for b in range(256))       # every single byte is a token
    assert toks[-1] == b""                                      # EOS: id V - 1, no bytes
    multi = toks[256:-1]
    assert min(map(len, multi)) == lo and max(map(len, multi)) == hi
    assert len(set(toks)) == w.V                                # token strings are distinct


def test_sets(wl):
    cfg, w, strings, _ = wl
    if cfg in (1, 2):
        assert len(set(strings)) == len(strings)
        assert all(SNAKE.fullmatch(s) and 8 <= len(s) <= 32 for s in strings)
    elif cfg in (3, 4):
        pat = CODES3 if cfg == 3 else CODES4
        assert len(set(strings)) == len(strings)
        assert all(pat.fullmatch(s) for s in strings)
        # categories (letter + 2 digits) are Zipf-skewed: a few hold many codes
        cats = np.unique([s[:3] for s in strings], return_counts=True)[1]
        assert cats.max() >= 10 * np.median(cats)
    else:
        idx = w.set_index
        assert len(idx) == 257 and idx[0] == 0 and idx[-1] == len(strings)
        ks = np.diff(idx)
        assert ks.min() >= 300 and ks.max() <= 2000
        pool = set(W.tool_names(5, 50000, 2000))
        for r in range(256):
            req = strings[idx[r]:idx[r + 1]]
            assert len(set(req)) == len(req), r
        assert set(strings) <= pool
        assert all(SNAKE.fullmatch(s) and 8 <= len(s) <= 32 for s in set(strings))


def test_tokens_follow_the_set_alphabet(wl):
    """The code vocabularies carry runs of [A-Z0-9] (20 % of the multi-byte
    tokens); the tool vocabularies draw 30 % of them from stem words."""
    cfg, w, _, toks = wl
    multi = toks[256:-1]
    if cfg == 3:
        runs = sum(1 for t in multi if re.fullmatch(rb"[A-Z0-9]{2,4}", t))
        assert runs >= 0.2 * len(multi)
    if cfg == 1:
        stems = W.tool_stems(0, 40)
        inside = sum(1 for t in multi[:2000] if any(t in s for s in stems))
        assert inside >= 0.25 * 2000


def test_node_counts_quoted_by_the_measurements(wl):
    """The node counts recorded with the results (host builder, no GPU)."""
    from paper_2608_12574_gb300 import _build
    from paper_2608_12574_gb300 import triemask as T
    _build.build()
    cfg, w, _, _ = wl
    want = {1: 1384, 2: 11506, 3: 23090, 4: 111296, 5: 4765457}[cfg]
    h = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index) if cfg == 5 \
        else T.trie_build(w.set_bytes, w.set_offsets)
    assert h.num_nodes == want
    h.destroy()


@pytest.mark.parametrize("cfg", [1, 3])
def test_logits_scale_and_seed(cfg):
    import torch
    w = W.config(cfg)
    x = W.logits(w, 0)
    assert tuple(x.shape) == (w.batch, w.V)
    assert x.dtype == (torch.float32 if w.dtype == "f32" else torch.bfloat16)
    assert abs(float(x.float().std()) - w.logit_std) < 0.02 * w.logit_std
    assert abs(float(x.float().mean())) < 0.02 * w.logit_std
    assert torch.equal(x, W.logits(w, 0))                      # seeded per step
    assert not torch.equal(x, W.logits(w, 1))
