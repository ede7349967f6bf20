"""GPU parity of the embedding tail (Sec. 4.3: masked mean pool of hidden
states, L2 normalisation, cast to the index dtype) against the fp64 oracle.
A bf16 output must be a correct rounding of a value within 2e-6 of the exact
result (the kernel accumulates in fp32); an fp32 output must lie within 2e-6."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08340_gb300 import workloads
from paper_2608_08340_gb300.index import Index, embed_pool

from _golden import load
from _gpu import check_dense, dev_tensor

pytestmark = pytest.mark.gpu

ERR = 2e-6


def _bf16_ok(got_bits, exact):
    got = oracle.bf16_to_f32(got_bits).astype(np.float64)
    # half a bf16 ulp of the exact value (8 bits of mantissa), plus the fp32 error
    ulp = np.where(exact != 0, 2.0 ** (np.floor(np.log2(np.abs(exact) + 1e-300)) - 7), 2.0 ** -133)
    return np.abs(got - exact) <= 0.5 * ulp + ERR


def test_embed_pool_golden_padded_to_eight_dims():
    g = load("embed_pool_2tok.json")
    h = np.zeros((3, 2, 8), np.float32)
    h[:, :, :2] = np.array(g["hidden"], np.float32)
    out = embed_pool(torch.from_numpy(h).cuda(), torch.tensor(g["mask"], dtype=torch.uint8).cuda())
    bits = out.view(torch.int16).cpu().numpy().view(np.uint16)
    assert bits[:, :2].tolist() == g["bf16_bits"]
    assert (bits[:, 2:] == 0).all()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("dim", [768, 4096, 136])
@pytest.mark.parametrize("out_dtype", [torch.bfloat16, torch.float32])
def test_embed_pool_matches_oracle(dtype, dim, out_dtype):
    rng = np.random.default_rng(dim + (dtype == "bf16"))
    b, t = 37, 50
    h = rng.standard_normal((b, t, dim)).astype(np.float32)
    lens = rng.integers(1, t + 1, b)
    mask = (np.arange(t)[None, :] < lens[:, None]).astype(np.uint8)
    mask[3] = 0                                            # a row with no real token
    mask[5] = (rng.random(t) < 0.3)                        # a row with holes
    h_in = oracle.round_bf16(h) if dtype == "bf16" else h
    exact = oracle.embed_pool(h_in, mask)
    out = embed_pool(dev_tensor(h_in), torch.from_numpy(mask).cuda(), out_dtype)
    torch.cuda.synchronize()
    if out_dtype == torch.bfloat16:
        bits = out.view(torch.int16).cpu().numpy().view(np.uint16)
        ok = _bf16_ok(bits, exact)
        assert ok.all(), f"{(~ok).sum()} of {ok.size} values off"
    else:
        np.testing.assert_allclose(out.cpu().numpy(), exact, rtol=0, atol=ERR)
    assert (out[3] == 0).all()


def test_embed_pool_feeds_the_search():
    w = workloads.config(1, n=8000, batch=4)
    rng = np.random.default_rng(11)
    h = oracle.round_bf16(rng.standard_normal((64, 20, w.d)).astype(np.float32))
    mask = np.ones((64, 20), np.uint8)
    mask[:, 15:] = 0
    Q = embed_pool(dev_tensor(h), torch.from_numpy(mask).cuda())
    idx = Index(dev_tensor(w.E_data))
    ids, sc = idx.search(Q, 10)
    q_bits = Q.view(torch.int16).cpu().numpy().view(np.uint16)
    check_dense(ids, sc, w.E_data, q_bits, 10, "pooled queries")


def test_embed_pool_argument_errors():
    h = torch.zeros((2, 3, 12), dtype=torch.bfloat16, device="cuda")       # dim not % 8
    with pytest.raises(RuntimeError):
        embed_pool(h, torch.ones((2, 3), dtype=torch.uint8, device="cuda"))
    h = torch.zeros((2, 3, 16), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ValueError):
        embed_pool(h, torch.ones((2, 4), dtype=torch.uint8, device="cuda"))
