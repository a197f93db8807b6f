"""Host-side pieces of the end-to-end decoder (Algorithm 1), on the CPU.

* donor token sequences follow Table 1's structure: the scaffold is kept,
  BLANK fills the content with one filler token, SAME_ALGO / DIFF_ALGO
  replace the ladder's fractions (0.1 / 0.5) of content positions, ZERO has
  no tokens;
* RoPE preserves norms and makes q . k depend only on the position offset;
* prefill is causal: a position's K and V do not depend on later tokens.
"""
import math

import pytest
import torch

from paper_2605_30574_gb300.model import RandomDecoder, donor_tokens, tiny_dims
from paper_2605_30574_gb300.synth import workloads as W


@pytest.fixture(scope="module")
def model():
    return RandomDecoder(tiny_dims(), seed=0, device="cpu")


def test_donor_tokens_follow_table1():
    g = torch.Generator()
    g.manual_seed(3)
    vocab, Tp, head, tail, filler = 50000, 4096, 24, 12, 7
    prompt = torch.randint(0, vocab, (Tp,), generator=g)
    content = slice(head, Tp - tail)
    n = Tp - head - tail
    assert donor_tokens(prompt, W.ZERO, g, vocab, head, tail, filler) is None
    for kind in (W.BLANK, W.SAME_ALGO, W.DIFF_ALGO, W.DIFF_FAMILY):
        d = donor_tokens(prompt, kind, g, vocab, head, tail, filler)
        assert d.shape == prompt.shape
        assert torch.equal(d[:head], prompt[:head]) and torch.equal(d[Tp - tail:], prompt[Tp - tail:])
    blank = donor_tokens(prompt, W.BLANK, g, vocab, head, tail, filler)
    assert bool((blank[content] == filler).all())
    for kind, p in ((W.SAME_ALGO, 0.1), (W.DIFF_ALGO, 0.5)):
        d = donor_tokens(prompt, kind, g, vocab, head, tail, filler)
        changed = int((d[content] != prompt[content]).sum())
        # binomial(n, p) within 5 standard deviations (a replaced token equals
        # the old one with probability 1 / vocab)
        assert abs(changed - n * p) < 5 * math.sqrt(n * p * (1 - p)) + 2, (kind, changed)
    fam = donor_tokens(prompt, W.DIFF_FAMILY, g, vocab, head, tail, filler)
    assert int((fam[content] != prompt[content]).sum()) > n - 10


def test_rope_is_a_relative_rotation(model):
    g = torch.Generator()
    g.manual_seed(1)
    d = model.dims.head_dim
    q = torch.randn(1, 1, d, generator=g)
    k = torch.randn(1, 1, d, generator=g)
    for m, n, c in ((5, 2, 100), (0, 31, 7), (400, 3, 1000)):
        qm, kn = model.rope(q, torch.tensor([m])), model.rope(k, torch.tensor([n]))
        assert torch.allclose(qm.norm(), q.norm(), rtol=1e-5)
        a = (qm * kn).sum()
        b = (model.rope(q, torch.tensor([m + c])) * model.rope(k, torch.tensor([n + c]))).sum()
        assert torch.allclose(a, b, rtol=1e-4, atol=1e-4), (m, n, c)


def test_prefill_is_causal(model):
    dims = model.dims
    g = torch.Generator()
    g.manual_seed(2)
    Tp = 24
    toks = torch.randint(0, dims.vocab, (Tp,), generator=g)
    alt = toks.clone()
    alt[-1] = (alt[-1] + 1) % dims.vocab
    shape = (dims.num_layers, dims.num_kv_heads, Tp, dims.head_dim)
    k1, v1, k2, v2 = (torch.empty(shape, dtype=torch.bfloat16) for _ in range(4))
    l1 = model.prefill(toks, k1, v1)
    l2 = model.prefill(alt, k2, v2)
    assert torch.equal(k1[:, :, :-1], k2[:, :, :-1]) and torch.equal(v1[:, :, :-1], v2[:, :, :-1])
    assert not torch.equal(k1[:, :, -1], k2[:, :, -1])
    assert not torch.equal(l1, l2)
