"""The Python binding's argument checks, on CPU.

Every wrapper validates shapes, dtypes and devices before it calls into the
library, so these checks run without a GPU: a logits tensor that is not
[B, V], not float32 / bfloat16 or not on a CUDA device, state and token
arrays whose length is not B, and vocabulary offsets of the wrong length are
refused with a Python exception and never reach the C ABI.
"""
from __future__ import annotations

import numpy as np
import pytest

from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W


@pytest.fixture(scope="module")
def handles():
    from paper_2608_12574_gb300 import _build
    _build.build()
    sb, so = W.pack([b"ab", b"ac"])
    h = T.trie_build(sb, so)
    f = T.fmt_build(W.format_classes("##-##"))
    yield h, f
    h.destroy()
    f.destroy()


def _t(shape, dtype="float32"):
    import torch
    return torch.zeros(shape, dtype=getattr(torch, dtype))


def _calls(h, f):
    """(name, call(logits, states, tokens, states_out)) of every masking wrapper."""
    return [
        ("trie_apply_mask", lambda lg, st, tk, so: T.trie_apply_mask(h, lg, st)),
        ("trie_apply_lists", lambda lg, st, tk, so: T.trie_apply_lists(h, lg, st)),
        ("trie_lazy_apply", lambda lg, st, tk, so: T.trie_lazy_apply(h, lg, st)),
        ("fmt_apply_mask", lambda lg, st, tk, so: T.fmt_apply_mask(f, lg, st)),
        ("trie_advance_apply", lambda lg, st, tk, so: T.trie_advance_apply(h, st, tk, so, lg)),
        ("trie_lazy_advance_apply", lambda lg, st, tk, so: T.trie_lazy_advance_apply(h, st, tk, so, lg)),
        ("trie_advance_apply_lists", lambda lg, st, tk, so: T.trie_advance_apply_lists(h, st, tk, so, lg)),
    ]


def test_masking_wrappers_check_their_arguments(handles):
    h, f = handles
    B, V = 3, 40
    st, tk, so = _t(B, "int32"), _t(B, "int32"), _t(B, "int32")
    for name, call in _calls(h, f):
        with pytest.raises(ValueError, match=r"\[B, V\]"):
            call(_t(B * V), st, tk, so)
        with pytest.raises(TypeError, match="float32 or bfloat16"):
            call(_t((B, V), "float16"), st, tk, so)
        with pytest.raises(ValueError, match="B entries"):
            call(_t((B, V)), _t(B + 1, "int32"), tk, so)
        with pytest.raises(TypeError, match="CUDA tensor"):        # host memory never reaches the kernels
            call(_t((B, V)), st, tk, so)
        with pytest.raises(TypeError, match="CUDA tensor"):
            call(_t((B, V), "bfloat16"), st, tk, so)
    for name, call in _calls(h, f)[4:]:                            # the advancing forms check the tokens too
        with pytest.raises(ValueError, match="B entries"):
            call(_t((B, V)), st, _t(B - 1, "int32"), so)
        with pytest.raises(ValueError, match="B entries"):
            call(_t((B, V)), st, tk, _t(B + 2, "int32"))


def test_other_wrappers_check_their_arguments(handles):
    h, f = handles
    vb, vo = W.pack([b"a", b"b", b""])
    with pytest.raises(ValueError, match="V\\+1"):
        T.trie_compile_masks(h, vb, vo, 4, _t((3, 1), "int32"))
    with pytest.raises(ValueError, match="V\\+1"):
        T.trie_compile_masks_noalloc(h, vb, vo, 4, _t((3, 1), "int32"))
    with pytest.raises(ValueError, match="V\\+1"):
        T.trie_compile_lists(h, vb, vo, 2)
    with pytest.raises(ValueError, match="V\\+1"):
        T.trie_lazy_init(h, vb, vo, 5, 8, 8)
    with pytest.raises(ValueError, match="V\\+1"):
        T.fmt_compile_masks(f, vb, vo, 2, _t((6, 1), "int32"))
    with pytest.raises(TypeError, match="CUDA tensor"):
        T.trie_compile_masks(h, vb, vo, 3, _t((h.num_nodes, 1), "int32"))
    with pytest.raises(ValueError, match="differ in length"):
        T.trie_advance(h, _t(2, "int32"), _t(3, "int32"))
    with pytest.raises(ValueError, match="differ in length"):
        T.fmt_advance(f, _t(2, "int32"), _t(3, "int32"))
    with pytest.raises(TypeError, match="CUDA tensor"):
        T.trie_advance(h, _t(2, "int32"), _t(2, "int32"))
    assert T.mask_words(1) == 1 and T.mask_words(32) == 1 and T.mask_words(33) == 2
    assert np.array_equal(h.roots(), [0])


def test_vocab_wrappers_check_their_arguments(handles):
    h, f = handles
    vb, vo = W.pack([b"a", b"b", b""])
    with pytest.raises(ValueError, match="V\\+1"):
        T.trie_vocab_create(vb, vo, 4)
    for bad in (None, "vocab", T.Vocab(None, 0)):
        with pytest.raises(ValueError, match="live Vocab"):
            T.trie_compile_lists_vocab(h, bad)
        with pytest.raises(ValueError, match="live Vocab"):
            T.trie_compile_masks_vocab(h, bad, _t((3, 1), "int32"))
