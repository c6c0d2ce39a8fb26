"""GPU parity of trie_advance_apply (advance, then mask the next logits, in one
launch) and of the compile-filled transition table, against the CPU oracle."""
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


def _bits(t):
    import torch
    t = t.cpu().contiguous()
    if t.dtype == torch.float32:
        return t.view(torch.int32).numpy().view(np.uint32)
    return t.view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_fused_decode_loop(cuda, cfg):
    """apply(step 0), then advance_apply for every later step, greedy argmax in
    between: masked logits, tokens and states equal the oracle's at every step."""
    import torch
    w = W.config(cfg)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    m = T.alloc_mask(h, w.V, cuda)
    T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, m)
    logits = [W.logits(w, s, device="cuda") for s in range(w.steps)]
    bufs = [torch.zeros(w.batch, dtype=torch.int32, device=cuda) for _ in range(2)]
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    got = []
    tok = None
    for t in range(w.steps):
        x = logits[t].clone()
        if t == 0:
            T.trie_apply_mask(h, x, bufs[0])
        else:
            T.trie_advance_apply(h, bufs[(t - 1) % 2], tok, bufs[t % 2], x, err)
        tok = torch.argmax(x, dim=1).to(torch.int32)
        got.append((x, tok.cpu().numpy(), bufs[t % 2].cpu().numpy().copy()))
    final = bufs[(w.steps - 1) % 2].clone()
    T.trie_advance(h, final, tok, err)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    masked, toks, sts, oerr = oracle.decode(ot, ov, (_bits(lg) for lg in logits), np.zeros(w.batch, np.int32))
    for t in range(w.steps):
        assert np.array_equal(_bits(got[t][0]), masked[t]), t
        assert np.array_equal(got[t][1], toks[t]), t
        if t > 0:
            assert np.array_equal(got[t][2], sts[t - 1]), t   # states the step was masked with
    assert np.array_equal(final.cpu().numpy(), sts[-1])
    assert int(err.item()) == oerr == 0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("seed", range(6))
def test_fused_random(cuda, dtype, seed):
    """Random (also invalid) states and tokens, random logit bits; V aligned
    (one fused launch) and unaligned (the two kernels in sequence)."""
    import torch
    strings, toks = random_case(4000 + seed)
    V = len(toks)
    sb, so = W.pack(strings)
    vb, vo = W.pack(toks)
    h = T.trie_build(sb, so)
    m = T.alloc_mask(h, V, cuda)
    T.trie_compile_masks(h, vb, vo, V, m)
    ot, ov = oracle.Trie(sb, so), oracle.Vocab(vb, vo)
    r = np.random.default_rng(seed)
    B = 300
    n = ot.num_nodes
    states = r.choice(np.array([-1, -2, n, -5] + list(range(n)) * 4, np.int32), B)
    tokens = r.choice(np.array([-1, V, V - 1] + list(range(V)) * 3, np.int32), B)
    want_states, werr = oracle.advance(ot, ov, states, tokens)
    if dtype == "f32":
        raw = r.integers(0, 2**32, (B, V), dtype=np.uint64).astype(np.uint32)
        x = torch.from_numpy(raw.view(np.int32)).view(torch.float32).to(cuda)
    else:
        raw = r.integers(0, 2**16, (B, V), dtype=np.uint32).astype(np.uint16)
        x = torch.from_numpy(raw.view(np.int16)).view(torch.bfloat16).to(cuda)
    want_logits = oracle.apply(ot, ov, raw, want_states)
    s_in = torch.as_tensor(states, device=cuda)
    s_out = torch.zeros_like(s_in)
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    T.trie_advance_apply(h, s_in, torch.as_tensor(tokens, device=cuda), s_out, x, err)
    assert np.array_equal(s_out.cpu().numpy(), want_states)
    assert int(err.item()) == werr
    assert np.array_equal(s_in.cpu().numpy(), states)   # the input states are not touched
    assert np.array_equal(_bits(x), want_logits)


def test_fused_errors(cuda):
    import torch
    sb, so = W.pack([b"ab"])
    h = T.trie_build(sb, so)
    s = torch.zeros(2, dtype=torch.int32, device=cuda)
    x = torch.zeros((2, 4), device=cuda)
    with pytest.raises(T.TrieError):          # before any compile
        T.trie_advance_apply(h, s, s.clone(), torch.zeros_like(s), x)
    vb, vo = W.pack([b"a", b"b", b"ab", b""])
    m = T.alloc_mask(h, 4, cuda)
    T.trie_compile_masks(h, vb, vo, 4, m)
    with pytest.raises(T.TrieError):          # in place
        T.trie_advance_apply(h, s, s.clone(), s, x)
    with pytest.raises(T.TrieError):          # V differs
        T.trie_advance_apply(h, s, s.clone(), torch.zeros_like(s), torch.zeros((2, 5), device=cuda))


def test_transitions_follow_the_vocabulary(cuda):
    """A handle recompiled with another vocabulary (dense or lists) must advance
    by the new vocabulary's bytes: no transition of the old one survives."""
    import torch
    w = W.config(1)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    r = np.random.default_rng(3)
    for k, seed in enumerate((0, 11, 0, 11)):
        spec = W.VocabSpec(V=3000, max_len=12, substr_frac=0.5, run_frac=0.0, run_len=(2, 4),
                           upper=False, mixed=False)
        vb, vo = W.byte_vocab(seed, spec, substr_src=W.tool_stems(0, 40))
        ov = oracle.Vocab(vb, vo)
        if k % 2 == 0:
            T.trie_compile_masks(h, vb, vo, 3000, T.alloc_mask(h, 3000, cuda))
        else:
            T.trie_compile_lists(h, vb, vo, 3000)
        # valid moves (from the oracle's masks) and random ones
        rows = r.integers(0, ot.num_nodes, 400).astype(np.int32)
        mk = oracle.mask_rows(ot, ov, rows)
        toks = []
        for i in range(len(rows)):
            allowed = np.nonzero(np.unpackbits(mk[i].view(np.uint8), bitorder="little")[:3000])[0]
            toks.append(int(r.choice(allowed)) if len(allowed) and i % 3 else int(r.integers(0, 3000)))
        toks = np.array(toks, np.int32)
        want, _ = oracle.advance(ot, ov, rows, toks)
        st = torch.as_tensor(rows, device=cuda)
        T.trie_advance(h, st, torch.as_tensor(toks, device=cuda))
        assert np.array_equal(st.cpu().numpy(), want), k


def test_fused_decode_loop_largest_workload_sampled(cuda):
    """K = 74,719 codes, V = 262,144, B = 256, fp32, 16 steps, in the bench's
    launch configuration (step 0 apply, then one advance + apply launch per
    step): every state each step against the oracle's advance by the same
    tokens, and on 8 sampled requests per step the masked logits and the
    greedy token against the oracle's (the oracle would take minutes for all
    256 x 262,144 logits of 16 steps)."""
    import torch
    w = W.config(4)
    h = T.trie_build(w.set_bytes, w.set_offsets)
    m = T.alloc_mask(h, w.V, cuda)
    T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, m)
    ot = oracle.Trie(w.set_bytes, w.set_offsets)
    ov = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    r = np.random.default_rng(4)
    bufs = [torch.zeros(w.batch, dtype=torch.int32, device=cuda) for _ in range(2)]
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    ost = np.zeros(w.batch, np.int32)
    tok = None
    for t in range(w.steps):
        lg = W.logits(w, t, device="cuda")
        x = lg.clone()
        if t == 0:
            T.trie_apply_mask(h, x, bufs[0])
        else:
            T.trie_advance_apply(h, bufs[(t - 1) % 2], tok, bufs[t % 2], x, err)
            ost, _ = oracle.advance(ot, ov, ost, tok.cpu().numpy())
        assert np.array_equal(bufs[t % 2].cpu().numpy(), ost), f"states differ at step {t}"
        tok = torch.argmax(x, dim=1).to(torch.int32)
        rows = np.sort(r.choice(w.batch, 8, replace=False))
        raw = _bits(lg[torch.as_tensor(rows, device=cuda)])
        want = oracle.apply(ot, ov, raw, ost[rows])
        assert np.array_equal(_bits(x[torch.as_tensor(rows, device=cuda)]), want), f"logits differ at step {t}"
        assert np.array_equal(tok.cpu().numpy()[rows], oracle.argmax(want)), f"tokens differ at step {t}"
    assert int(err.item()) == 0
