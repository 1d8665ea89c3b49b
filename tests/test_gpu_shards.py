"""Parameter-sharded commits on one GPU, against one handle over all P, bit for bit.

Every step of a commit is elementwise (Algorithm 1 applies Psi_GEM with an elementwise
product), so a parameter vector split into contiguous shards, each with its own handle,
commits the matching gradient slices with no exchange between shards.  Here the shards
are handles on the same GPU (one per rank of a sharded run); each commits its slice of
every gradient, and the concatenated theta, m and s must equal the single handle's bits.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_1805_08469_gb300 import gem
from paper_1805_08469_gb300._build import build_library

pytestmark = pytest.mark.gpu

ETA, MU, EPS = 0.01, 0.9, 1e-8


@pytest.fixture(scope="module", autouse=True)
def _setup():
    build_library()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    torch.cuda.set_device(0)


@pytest.mark.parametrize("P,world", [(1_000_003, 2), (1_000_003, 3), (100, 2), (33, 4)])
@pytest.mark.parametrize("mode,kappa", [(gem.GEM_MODE_GEM, 1.0), (gem.GEM_MODE_KAPPA_SQRT, 4.0),
                                        (gem.GEM_MODE_ADAPTIVE, 1.0)])
def test_shards_equal_one_handle(P, world, mode, kappa):
    n, T = 7, 260
    rng = np.random.default_rng(P + world)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    Pp = (P + 3) // 4 * 4
    grads = torch.zeros((T, Pp), device="cuda")
    grads[:, :P] = torch.from_numpy((0.1 * rng.standard_normal((T, P))).astype(np.float32)).cuda()
    order, _tau = oracle.schedule_uniform(P + world, n, T)
    order = order.tolist()
    ranges = [gem.gem_shard_range(P, world, r) for r in range(world)]
    assert ranges[0][0] == 0 and max(e for _b, e in ranges) == P
    for (b0, e0), (b1, _e1) in zip(ranges, ranges[1:]):
        assert e0 == b1 and (b0 % 32 == 0 or b0 == P)   # an empty trailing shard starts at P
    full = gem.Gem(P, n, ETA, MU, EPS)
    shards = [gem.Gem(e - b, n, ETA, MU, EPS) if e > b else None for b, e in ranges]
    try:
        for G, (b, e) in [(full, (0, P))] + list(zip(shards, ranges)):
            if G is None:
                continue
            G.set_mode(mode, kappa)
            G.set_theta(torch.from_numpy(theta0[b:e].copy()).cuda())
            # single commits, then batches of 200 and 60 (one launch each)
            for k in range(0, 20):
                G.commit(order[k], grads[k, b:e])
            G.commit_batch(order[20:220], [grads[k, b:e] for k in range(20, 220)])
            G.commit_batch(order[220:], [grads[k, b:e] for k in range(220, T)])
            G.sync()
        for G, (b, e) in zip(shards, ranges):
            if G is None:
                continue
            assert torch.equal(G.theta(), full.theta()[b:e])
            for w in range(n):
                assert torch.equal(G.moment(w), full.moment(w)[b:e])
                assert torch.equal(G.snapshot(w), full.snapshot(w)[b:e])
    finally:
        full.close()
        for G in shards:
            if G is not None:
                G.close()
