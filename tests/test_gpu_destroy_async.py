"""trie_destroy_async: a handle released right after its last queued kernel.

The work queued before the release must still run on the handle's device
memory and host arrays (the upload of a host-built trie reads the host arrays
from a kernel where the GPU reads host memory coherently), so every result is
checked after the stream is synchronised, over several handles built and
released in turn on one stream."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W

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


def test_release_after_queued_work(cuda):
    import torch
    w = W.config(1)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    want = oracle.mask_all(ot, ov)
    stream = torch.cuda.Stream(cuda)
    B = 4
    logits = [W.logits(w, i, device="cuda", batch=B) for i in range(6)]
    states = [torch.tensor([0, 1, 2, 3 + i], dtype=torch.int32, device=cuda) for i in range(6)]
    wants = []
    for i, x in enumerate(logits):
        bits = x.cpu().view(torch.int32).numpy().view(np.uint32).copy()
        masked, _, _, _ = oracle.decode(ot, ov, [bits], np.array([0, 1, 2, 3 + i], np.int32))
        wants.append(masked[0])
    masks = [torch.empty((ot.num_nodes, T.mask_words(w.V)), dtype=torch.int32, device=cuda) for _ in range(6)]
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for i in range(6):  # no synchronisation inside: each release follows its queued work
            h = T.trie_build(w.set_bytes, w.set_offsets)
            T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, masks[i], stream)
            T.trie_apply_mask(h, logits[i], states[i], stream)
            h.destroy_async(stream)
    stream.synchronize()
    for m, x, wx in zip(masks, logits, wants):
        assert np.array_equal(m.cpu().view(torch.int32).numpy().view(np.uint32), want)
        assert np.array_equal(x.cpu().view(torch.int32).numpy().view(np.uint32), wx)
