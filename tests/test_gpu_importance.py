"""Offline preparation on the GPU (Sec. 3.2): Eq. 10 importance scores
(qsvd_importance_scores) against oracle.rank (itself pinned to Eq. 9's
definition), and the cross-layer rank budget (qsvd_rank_budget) against
oracle.rank.allocate_ranks, bit for bit including its tie rule.

The scores are fp32 sums over the n columns of each gradient and the m rows
of each singular vector, in a fixed order: the same bits on every run, and
within 1e-4 of the largest score of the fp64 oracle on the same fp32 inputs.
"""
import numpy as np
import pytest
import torch

from gpu_util import dev, q
from oracle import rank

pytestmark = pytest.mark.gpu

f32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev())  # noqa: E731
r32 = lambda a: np.asarray(a, dtype=np.float32).astype(np.float64)  # noqa: E731


def _problem(N, m, n, k, seed):
    rng = np.random.default_rng(seed)
    U = rng.standard_normal((m, k)) / np.sqrt(m)
    s = np.sort(rng.uniform(0.1, 3.0, k))[::-1].copy()
    Vt = rng.standard_normal((k, n)) / np.sqrt(n)
    G = rng.standard_normal((N, m, n))
    return U, s, Vt, G


@pytest.mark.parametrize("N,m,n,k", [(1, 64, 32, 64), (3, 200, 150, 70), (2, 96, 300, 129),
                                     (2, 1024, 3072, 1024)])
def test_importance_scores_match_oracle(N, m, n, k):
    """Ragged tiles (128 singular values and 256 rows per tensor-core CTA, 64
    on the CUDA-core path that n = 150 takes), k > n and k < n, and a
    joint-QKV-like shape (n = 3m) with 4 row tiles."""
    U, s, Vt, G = _problem(N, m, n, k, seed=N * 1000 + m)
    got = q().qsvd_importance_scores(f32(U), f32(s), f32(Vt), f32(G)).cpu().numpy().astype(np.float64)
    q().qsvd_check()
    want = rank.importance_scores(r32(U), r32(s), r32(Vt), [r32(g) for g in G])
    np.testing.assert_allclose(got, want, rtol=1e-4, atol=1e-4 * want.max())


def test_importance_scores_bench_shape_sampled():
    """The 7B joint-QKV shape the bench times (m = 4096, n = 3 x 4096,
    k = 4096, one sample) on the tensor-core path; 96 singular values
    checked against the oracle (a score depends only on its own singular
    triplet and G, so the oracle runs on that subset)."""
    N, m, n, k = 1, 4096, 12288, 4096
    U, s, Vt, G = _problem(N, m, n, k, seed=11)
    got = q().qsvd_importance_scores(f32(U), f32(s), f32(Vt), f32(G)).cpu().numpy().astype(np.float64)
    q().qsvd_check()
    idx = np.unique(np.concatenate([np.arange(32), np.random.default_rng(5).choice(k, 64, replace=False)]))
    want = rank.importance_scores(r32(U[:, idx]), r32(s[idx]), r32(Vt[idx]), [r32(g) for g in G])
    np.testing.assert_allclose(got[idx], want, rtol=1e-4, atol=1e-4 * want.max())


def test_importance_scores_deterministic_and_budget_boundary():
    """Two calls give identical bits; and the rank budget taken from the GPU
    scores keeps the same singular values as the one taken from the oracle's,
    except for pairs whose scores lie within the tolerance of the boundary."""
    N, m, n, k = 1, 1024, 3072, 1024
    U, s, Vt, G = _problem(N, m, n, k, seed=77)
    lib = q()
    a = lib.qsvd_importance_scores(f32(U), f32(s), f32(Vt), f32(G))
    b = lib.qsvd_importance_scores(f32(U), f32(s), f32(Vt), f32(G))
    lib.qsvd_check()
    assert torch.equal(a, b)
    got = a.cpu().numpy().astype(np.float64)
    want = rank.importance_scores(r32(U), r32(s), r32(Vt), [r32(g) for g in G])
    budget = 300
    keep_gpu = set(rank.allocate_ranks([got], budget)[0])
    keep_ref = set(rank.allocate_ranks([want], budget)[0])
    boundary = np.sort(want)[::-1][budget - 1]
    tol = 1e-4 * want.max() + 1e-4 * boundary
    for i in keep_gpu ^ keep_ref:
        assert abs(want[i] - boundary) <= 2 * tol, (i, want[i], boundary)


def test_importance_argument_errors():
    lib = q()
    z = torch.zeros((4, 4), dtype=torch.float32, device=dev())
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_importance_scores(z, torch.zeros(4, device=dev()), z, torch.zeros((1, 4, 4), device=dev()),
                                   workspace=torch.zeros(4, dtype=torch.uint8, device=dev()))
    assert e.value.status == lib.QSVD_ENOSPC


def _keep_ref(per_layer, k):
    kept = rank.allocate_ranks(per_layer, k)
    out = []
    for scores, idx in zip(per_layer, kept):
        m = np.zeros(len(scores), dtype=np.uint8)
        m[idx] = 1
        out.append(m)
    return np.concatenate(out)


@pytest.mark.parametrize("k", [0, 1, 777, 4000, 6144])
def test_rank_budget_matches_oracle(k):
    """32 layers of 192 scores with many exact ties (scores drawn from a
    small set) and a run of equal scores across the boundary: the tie rule
    (lower layer, then lower index) decides which of them are kept."""
    rng = np.random.default_rng(k + 5)
    per_layer = [np.round(rng.exponential(1.0, 192), 1).astype(np.float32).astype(np.float64) for _ in range(32)]
    per_layer[7][:50] = per_layer[20][:50] = 0.5
    flat = np.concatenate(per_layer)
    keep = q().qsvd_rank_budget(f32(flat), k).cpu().numpy()
    q().qsvd_check()
    assert int(keep.sum()) == k
    np.testing.assert_array_equal(keep, _keep_ref(per_layer, k))


def test_rank_budget_all_equal_and_extremes():
    """All scores equal: the first k positions; zeros and very large scores;
    a layout with one huge layer (131072 values, 7B-like: 32 x 4096)."""
    lib = q()
    flat = np.full(1000, 2.5)
    np.testing.assert_array_equal(lib.qsvd_rank_budget(f32(flat), 333).cpu().numpy(), (np.arange(1000) < 333))
    rng = np.random.default_rng(3)
    per_layer = [rng.exponential(1.0, 4096) * 10.0 ** rng.integers(-30, 30) for _ in range(32)]
    per_layer[0][:10] = 0.0
    per_layer[1][:5] = 3.0e38
    per_layer = [p.astype(np.float32).astype(np.float64) for p in per_layer]
    for k in (1, 4096, 65536, 131071):
        keep = lib.qsvd_rank_budget(f32(np.concatenate(per_layer)), k).cpu().numpy()
        np.testing.assert_array_equal(keep, _keep_ref(per_layer, k))
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_rank_budget(f32(flat), 1001)
    assert e.value.status == lib.QSVD_EINVAL
