"""Top-K selection stage (moe_topk) on seeded fp32 logits, in particular rows
of more than 128 experts (eight lanes per token): indices bit-exact against
the oracle's selection of the same logits (ties to the lower expert index,
ordered by descending logit), probabilities within 1e-5, for K from 1 to 16
and token counts that leave a ragged last block."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import PROB_ABS, f64, i64

pytestmark = pytest.mark.gpu

CASES = [(E, K) for E in (64, 128, 136, 200, 256) for K in (1, 2, 8, 16) if K <= E]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("E,K", CASES, ids=[f"E{e}_K{k}" for e, k in CASES])
def test_topk_matches_oracle(E, K):
    from paper_2608_28511_gb300 import abi
    T = 1000
    w = synth.Workload(f"tk_{E}_{K}", S=T, GBS=1, D=64, E=E, K=K, F=64)
    g = torch.Generator().manual_seed(E * 31 + K)
    z = torch.randn(T, E, generator=g)
    z[::7, 5] = z[::7, 3]                       # exact ties: the lower expert index wins
    z[::11, : E // 2] = 0.25                    # a block of equal logits
    z[13] = 1.0                                 # a row of all-equal logits
    zd = z.cuda()
    idx = torch.empty(T, K, dtype=torch.int32, device="cuda")
    prob = torch.empty(T, K, device="cuda")
    abi.moe_topk(abi.MoeShape.from_workload(w), zd, idx, prob)
    torch.cuda.synchronize()
    idx_ref, prob_ref = O.top_k_route(z.double().numpy(), K)
    assert (i64(idx) == idx_ref).all()
    assert np.abs(f64(prob) - prob_ref).max() <= PROB_ABS
