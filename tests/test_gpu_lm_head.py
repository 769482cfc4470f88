"""ptd_lm_head_topk on the GPU against the oracle (the per-node logits of Alg. 1 step 2
and their top-k, Sec. 3.1 / 3.2).

The logits are fp32 sums of K = d_model bf16 products accumulated by the tensor cores in an
order of their own, so each returned value must equal the exact (float64) logit of its
token within the fp32 bound K * 2^-24 * sum_j |h_j w_j|, the j-th returned value must be
within that of the exact j-th largest, and the tokens must be exactly the oracle's wherever
the exact values are farther apart than twice the bound (a near tie may swap).  Exact ties
(duplicated weight rows) must keep the lower token first."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _inputs(rows, d, vocab, seed, h_stride=None, w_stride=None, dup=()):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    hs, ws = h_stride or d, w_stride or d
    hbuf = torch.randn((rows, hs), generator=g, device="cuda").to(torch.bfloat16)
    wbuf = (torch.randn((vocab, ws), generator=g, device="cuda") / d ** 0.5).to(torch.bfloat16)
    for a, b in dup:                                      # token b gets token a's weights
        wbuf[b] = wbuf[a]
    return hbuf[:, :d], wbuf[:, :d]


def _run(h, w, k):
    rows, vocab = h.shape[0], w.shape[0]
    ws = torch.empty(ptd.lm_head_workspace_size(rows, vocab), dtype=torch.uint8, device="cuda")
    idx = torch.full((rows, k), -7, dtype=torch.int32, device="cuda")
    val = torch.full((rows, k), float("nan"), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert ptd.lm_head_topk(h, w, k, idx, val, ws, st) == 2
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return idx.cpu().numpy(), val.cpu().numpy()


def _exact(h, w, rows):
    """float64 logits [len(rows), V] and their fp32 bounds, the weights taken in chunks."""
    h64 = h[list(rows)].float().cpu().double().numpy()
    d = h64.shape[1]
    ex, bd = [], []
    for i in range(0, w.shape[0], 16384):
        wc = w[i:i + 16384].float().cpu().double().numpy()
        ex.append(wc @ h64.T)
        bd.append(d * 2.0 ** -24 * (np.abs(wc) @ np.abs(h64).T))
    return np.concatenate(ex).T, np.concatenate(bd).T


def _check_rows(idx, val, exact_rows, bound_rows, k):
    for r in range(len(exact_rows)):
        exact, bound = exact_rows[r], bound_rows[r]
        gi, gv = idx[r], val[r]
        assert len(set(gi.tolist())) == k and gi.min() >= 0 and gi.max() < len(exact)
        assert np.all(np.diff(gv) <= 0)
        assert np.all(np.abs(gv - exact[gi]) <= bound[gi] + 1e-30)
        ref_i, ref_v = oracle.topk(exact, k)
        tol = 2 * bound.max()
        assert np.all(np.abs(gv - ref_v) <= tol)
        ext = np.sort(exact)[::-1][:k + 1]
        for j in range(k):                                 # well separated ranks are exact
            gap_up = ext[j - 1] - ext[j] if j > 0 else np.inf
            gap_down = ext[j] - ext[j + 1] if j + 1 < len(ext) else np.inf
            if min(gap_up, gap_down) > tol:
                assert gi[j] == ref_i[j], (r, j)


CASES = [
    # rows, d_model, vocab, k
    (63, 512, 10000, 4),      # the step's 63 nodes; a ragged last tile (10000 = 78 * 128 + 16)
    (1, 64, 200, 1),          # plain decoding: one row, one 64-column chunk
    (128, 1024, 32000, 8),    # a full 128-row tile
    (100, 256, 130, 16),      # two tiles, the second 2 tokens wide; k = 16
]


@pytest.mark.parametrize("rows,d,vocab,k", CASES)
def test_lm_head_topk_matches_oracle(rows, d, vocab, k):
    h, w = _inputs(rows, d, vocab, 81 + rows)
    idx, val = _run(h, w, k)
    _check_rows(idx, val, *_exact(h, w, range(rows)), k)


def test_strided_rows():
    h, w = _inputs(40, 256, 3000, 91, h_stride=256 + 64, w_stride=256 + 8)
    assert h.stride(0) == 320 and w.stride(0) == 264
    idx, val = _run(h, w, 4)
    _check_rows(idx, val, *_exact(h, w, range(40)), 4)


def test_exact_ties_keep_the_lower_token():
    """Token 4000's weights copied to tokens 17 and 2500: their logits are equal to the bit,
    so wherever they reach the top-k they appear in the order 17, 2500, 4000."""
    h, w = _inputs(16, 128, 5000, 92)
    w[4000] = h[0]                                         # the top token of node 0, by far
    w[17] = w[4000]
    w[2500] = w[4000]
    idx, val = _run(h, w, 6)
    for r in range(16):
        pos = [list(idx[r]).index(t) for t in (17, 2500, 4000) if t in idx[r]]
        assert pos == sorted(pos)
    assert list(idx[0][:3]) == [17, 2500, 4000] and val[0][0] == val[0][1] == val[0][2]


def test_llama3_lm_head_full_size_sampled_rows():
    """The Llama-3-8B-shaped head: 63 rows, d_model 4096, vocab 128256 (1.05 GB of
    weights); three rows checked against float64 logits over the whole vocabulary."""
    rows, d, vocab, k = 63, 4096, 128256, 4
    h, w = _inputs(rows, d, vocab, 93)
    idx, val = _run(h, w, k)
    sample = [0, 31, 62]
    _check_rows(idx[sample], val[sample], *_exact(h, w, sample), k)
