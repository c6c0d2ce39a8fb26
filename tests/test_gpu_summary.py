"""The dense compile's segment summary across compiles and CUDA graphs.

The probe of each compile tags the summary words it sets with the compile's
epoch and publishes that epoch on the device; the applies read the epoch at
run time and take a word with another tag as empty. These tests interleave
compiles with other vocabularies, graph replays of earlier compiles and
graphs that hold only applies, and check every masked logit against the
oracle's mask of the compile that ran last.
"""
from __future__ import annotations

import os

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W

pytestmark = pytest.mark.gpu
NCPU = os.cpu_count() or 1
V = 5000  # five 1,024-token segments per row


@pytest.fixture(scope="module")
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_12574_gb300 import _build
    _build.build()
    oracle.build()
    return torch.device("cuda:0")


def _vocab(seed):
    spec = W.VocabSpec(V=V, max_len=12, substr_frac=0.3, run_frac=0.0, run_len=(2, 4), upper=False, mixed=False)
    return W.byte_vocab(seed, spec, substr_src=W.tool_stems(0, 40))


def _bits16(t):
    import torch
    return t.cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _expected(want_mask, states, logits_bits):
    """Masked bf16 bits from the oracle's mask rows (EOS only for non-nodes)."""
    out = logits_bits.copy()
    n = want_mask.shape[0]
    v = np.arange(V)
    for b, s in enumerate(states):
        if 0 <= s < n:
            allowed = ((want_mask[s][v >> 5] >> (v & 31).astype(np.uint32)) & 1).astype(bool)
        else:
            allowed = v == V - 1
        out[b][~allowed] = np.uint16(0xFF80)
    return out


def _states(ot, B, seed):
    r = np.random.default_rng(seed)
    return r.choice(np.array([-1, -2] + list(range(ot.num_nodes)) * 3, np.int32), B)


def test_summary_follows_the_last_compile(cuda):
    """Compiles with vocabularies A, B, A on one handle and mask buffer, each
    followed by applies: the words B leaves untouched still carry A's tag and
    must read as empty."""
    import torch
    w = W.config(1)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    m = T.alloc_mask(h, V, cuda)
    B = 96
    logits = torch.randn(B, V, generator=torch.Generator().manual_seed(1)).to(torch.bfloat16)
    for i, seed in enumerate((0, 7, 0, 3)):
        vb, vo = _vocab(seed)
        T.trie_compile_masks(h, vb, vo, V, m)
        want = oracle.mask_all(ot, oracle.Vocab(vb, vo), nthreads=NCPU)
        assert np.array_equal(m.cpu().numpy().view(np.uint32), want)
        st = _states(ot, B, 10 + i)
        x = logits.to(cuda)
        T.trie_apply_mask(h, x, torch.tensor(st, device=cuda))
        assert np.array_equal(_bits16(x), _expected(want, st, _bits16(logits))), seed


def test_summary_with_graphs(cuda):
    """A graph of [compile A, apply] and a graph of applies alone, replayed
    between eager compiles with the same vocabulary (each a new epoch), then
    an eager compile with vocabulary B: every result against the oracle's
    mask of the compile that ran last. (Graphs are not replayed after the
    compile with B: captured work must not outlive a later compile of the
    handle with another vocabulary.)"""
    import torch
    w = W.config(1)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    (vba, voa), (vbb, vob) = _vocab(0), _vocab(7)
    want_a = oracle.mask_all(ot, oracle.Vocab(vba, voa), nthreads=NCPU)
    want_b = oracle.mask_all(ot, oracle.Vocab(vbb, vob), nthreads=NCPU)
    m = T.alloc_mask(h, V, cuda)
    B = 64
    src = torch.randn(B, V, generator=torch.Generator().manual_seed(2)).to(torch.bfloat16).to(cuda)
    x = torch.empty_like(src)
    st = _states(ot, B, 5)
    dst = torch.tensor(st, device=cuda)
    stream = torch.cuda.Stream(cuda)
    va, vb = T.trie_vocab_create(vba, voa, V), T.trie_vocab_create(vbb, vob, V)

    def compile_apply():
        x.copy_(src)
        T.trie_compile_masks_vocab(h, va, m, stream)
        T.trie_apply_mask(h, x, dst, stream)

    def apply_only():
        x.copy_(src)
        T.trie_apply_mask(h, x, dst, stream)

    g1, g2 = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        compile_apply()
        with torch.cuda.graph(g1, stream=stream):
            compile_apply()
        with torch.cuda.graph(g2, stream=stream):
            apply_only()
    stream.synchronize()
    exp_a = _expected(want_a, st, _bits16(src))
    exp_b = _expected(want_b, st, _bits16(src))
    with torch.cuda.stream(stream):
        g1.replay()
    stream.synchronize()
    assert np.array_equal(_bits16(x), exp_a)
    with torch.cuda.stream(stream):
        T.trie_compile_masks_vocab(h, va, m, stream)  # A eagerly: a new epoch, the same bits
        g2.replay()  # applies captured before: they read the epoch now current
    stream.synchronize()
    assert np.array_equal(_bits16(x), exp_a)
    with torch.cuda.stream(stream):
        g1.replay()  # the graph's own epoch again, after the eager one
        g2.replay()
        g1.replay()
    stream.synchronize()
    assert np.array_equal(_bits16(x), exp_a)
    with torch.cuda.stream(stream):
        T.trie_compile_masks_vocab(h, vb, m, stream)  # B: the words only A set keep older tags
        apply_only()
    stream.synchronize()
    assert np.array_equal(_bits16(x), exp_b)
    assert np.array_equal(m.cpu().numpy().view(np.uint32), want_b)
