"""GPU parity of the character-position masks for fixed formats (App. K)
through the C ABI: masks, positions and masked logits bit-identical to the
oracle's, on small random formats (exhaustive), the four formats of the
paper's comparison with the workloads' vocabularies (tokens up to 24 bytes),
and a greedy decode that must always produce a string of the format.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W
from pins import fmt_bitmaps, fmt_case

pytestmark = pytest.mark.gpu


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


def _compile(cuda, classes, vb, vo, V):
    f = T.fmt_build(classes)
    m = T.fmt_alloc_mask(f, V, cuda)
    m.fill_(-1)  # every word must be written
    T.fmt_compile_masks(f, vb, vo, V, m)
    return f, m


@pytest.mark.parametrize("seed", range(40))
def test_fmt_small_random_exhaustive(cuda, seed):
    import torch
    cls, toks = fmt_case(9000 + seed)
    vb, vo = W.pack(toks)
    V = len(toks)
    c = fmt_bitmaps(cls)
    f, m = _compile(cuda, c, vb, vo, V)
    of, ov = oracle.Format(c), oracle.Vocab(vb, vo)
    assert np.array_equal(_np_u32(m), of.mask_all(ov))
    r = np.random.default_rng(seed)
    L = len(cls)
    states = r.choice(np.array([-1, -2, L + 1, -5] + list(range(L + 1)) * 4, np.int32), 300)
    tokens = r.choice(np.array([-1, V, V - 1] + list(range(V)) * 3, np.int32), 300)
    want, werr = of.advance(ov, states, tokens)
    ds = torch.as_tensor(states, device=cuda).clone()
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    T.fmt_advance(f, ds, torch.as_tensor(tokens, device=cuda), err)
    assert np.array_equal(ds.cpu().numpy(), want) and int(err.item()) == werr


@pytest.mark.parametrize("name", list(W.FORMATS))
@pytest.mark.parametrize("cfg", [1, 3, 4])
def test_fmt_paper_formats(cuda, name, cfg):
    """Every position of the format against the oracle, with a workload
    vocabulary (cfg 4's tokens reach 24 bytes, past one 16-byte chunk)."""
    w = W.config(cfg)
    c = W.format_classes(W.FORMATS[name])
    f, m = _compile(cuda, c, w.vocab_bytes, w.vocab_offsets, w.V)
    want = oracle.Format(c).mask_all(oracle.Vocab(w.vocab_bytes, w.vocab_offsets))
    assert np.array_equal(_np_u32(m), want)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_fmt_greedy_decode_is_valid(cuda, dtype):
    """apply -> greedy -> advance until EOS: logits, tokens and positions
    equal the oracle's at every step, and every finished request spells a
    string of the format. Tokens of the date format: digits and runs of
    digits, dashes, and a few longer pieces."""
    import torch
    digits = [str(i).encode() for i in range(10)]
    toks = (digits + [a + b for a in digits for b in digits] + [b"-", b"20", b"2024", b"-0", b"-1", b"1-",
            b"12-", b"-12-", b"x", b"2024-05-17", b"ab", b"0000-00-00"] + [b""])
    vb, vo = W.pack(toks)
    V = len(toks)
    c = W.format_classes(W.FORMATS["YYYY-MM-DD"])
    f, m = _compile(cuda, c, vb, vo, V)
    of, ov = oracle.Format(c), oracle.Vocab(vb, vo)
    B = 64
    g = torch.Generator(device="cpu").manual_seed(5)
    st = torch.zeros(B, dtype=torch.int32, device=cuda)
    ost = np.zeros(B, np.int32)
    out = [[] for _ in range(B)]
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    for step in range(12):
        x = (torch.randn((B, V), generator=g) * 2).to(tdt).to(cuda)
        xb = _bits(x)
        T.fmt_apply_mask(f, x, st)
        want = of.apply(ov, xb, ost)
        assert np.array_equal(_bits(x), want), f"step {step}"
        tok = torch.argmax(x.float(), dim=1).to(torch.int32)
        otok = oracle.argmax(want)
        assert np.array_equal(tok.cpu().numpy(), otok)
        T.fmt_advance(f, st, tok)
        ost, _ = of.advance(ov, ost, otok)
        assert np.array_equal(st.cpu().numpy(), ost)
        for b in range(B):
            if otok[b] != V - 1:
                out[b].append(toks[otok[b]])
    done = [b for b in range(B) if ost[b] == oracle.FINISHED]
    assert done and all(ost[b] in (oracle.FINISHED,) or 0 <= ost[b] <= 10 for b in range(B))
    import re
    for b in done:
        assert re.fullmatch(rb"[0-9]{4}-[0-9]{2}-[0-9]{2}", b"".join(out[b])), b"".join(out[b])


def test_fmt_edge_cases(cuda):
    import torch
    toks = [b"a", b"ab", b"", b"abc", b""]
    vb, vo = W.pack(toks)
    V = len(toks)
    # L = 0: only EOS, at position 0
    f, m = _compile(cuda, np.zeros((0, 32), np.uint8), vb, vo, V)
    assert _np_u32(m).tolist() == [[1 << (V - 1)]]
    # a token longer than the format is never allowed
    c = fmt_bitmaps([[ord("a")], [ord("b")]])
    f, m = _compile(cuda, c, vb, vo, V)
    assert np.array_equal(_np_u32(m), oracle.Format(c).mask_all(oracle.Vocab(vb, vo)))
    # V mismatch, B = 0
    with pytest.raises(T.TrieError):
        T.fmt_apply_mask(f, torch.zeros((1, V + 1), device=cuda), torch.zeros(1, dtype=torch.int32, device=cuda))
    e = torch.empty(0, dtype=torch.int32, device=cuda)
    T.fmt_advance(f, e, e)
    T.fmt_apply_mask(f, torch.empty((0, V), device=cuda), e)


@pytest.mark.parametrize("L", [63, 64, 200])
def test_fmt_long_formats(cuda, L):
    """Formats at and past 63 positions (the 64-bit position-set path ends
    at 63), tokens up to 40 bytes."""
    r = np.random.default_rng(L)
    alpha = [ord(c) for c in "0123456789abc-:"]
    cls = [sorted(r.choice(alpha, r.integers(1, 6), replace=False).tolist()) for _ in range(L)]
    toks = [bytes([c]) for c in alpha]
    for _ in range(700):
        n = int(r.integers(2, 41))
        toks.append(bytes(r.choice(alpha, n).tolist()))
    # tokens cut from strings of the format, so that long ones fit somewhere
    for _ in range(300):
        p0 = int(r.integers(0, L))
        n = int(r.integers(1, min(40, L - p0) + 1))
        toks.append(bytes(int(r.choice(cls[p0 + i])) for i in range(n)))
    toks.append(b"")
    vb, vo = W.pack(toks)
    V = len(toks)
    c = fmt_bitmaps(cls)
    f, m = _compile(cuda, c, vb, vo, V)
    want = oracle.Format(c).mask_all(oracle.Vocab(vb, vo))
    assert want[:, :].sum() > 0
    assert np.array_equal(_np_u32(m), want)
