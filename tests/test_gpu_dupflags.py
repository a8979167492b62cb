"""The repeated-hash flags (route_dup_flags) through the C ABI against a
direct check on the host: random hashes in the route_hash_blocks layout with
planted repeats, ragged prompt lengths and start offsets, prompts longer than
max_blocks, the largest max_blocks, values shared across requests (not a
repeat), and rejected arguments.  Flags are compared bit-exactly."""
import numpy as np
import pytest

from paper_2606_17081_gb300 import routesim as rs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


def _case(n, max_blocks, seed, long_frac=0.05, plant_frac=0.3, share_frac=0.2):
    rng = np.random.default_rng(seed)
    nb = rng.integers(0, max_blocks + 1, n)
    longer = rng.random(n) < long_frac
    nb[longer] = max_blocks + 1 + rng.integers(0, 40, int(longer.sum()))
    lens = nb * 16 + rng.integers(0, 16, n)          # a partial tail block is no block
    o0 = int(rng.integers(0, 64))
    offsets = np.concatenate([[o0], o0 + np.cumsum(lens)]).astype(np.int64)
    nh = int(offsets[-1]) // 16 + 1
    h = rng.integers(2, np.iinfo(np.uint64).max, nh, dtype=np.uint64, endpoint=True)
    for i in range(n):
        b, k = int(offsets[i]) // 16, int(nb[i])
        if k >= 2 and rng.random() < plant_frac:
            a, c = sorted(rng.choice(k, 2, replace=False))
            if rng.random() < 0.3:
                a, c = 0, k - 1                            # the two ends
            h[b + c] = h[b + a]
        elif k >= 1 and i > 0 and nb[i - 1] >= 1 and rng.random() < share_frac:
            pb = int(offsets[i - 1]) // 16                 # a value of the previous prompt
            h[b + int(rng.integers(0, k))] = h[pb + int(rng.integers(0, nb[i - 1]))]
    want = np.zeros(n, np.uint8)
    for i in range(n):
        b, k = int(offsets[i]) // 16, int(nb[i])
        if k > max_blocks:
            want[i] = 2
        elif len(set(h[b:b + k].tolist())) < k:
            want[i] = 1
    return offsets, h, want


def _run(offsets, h, n, max_blocks):
    ctx = rs.Context(W=2, K=64)
    hd = torch.from_numpy(h.view(np.int64)).cuda()
    od = torch.from_numpy(offsets).cuda()
    fl = torch.full((max(n, 1),), 0xAB, dtype=torch.uint8, device="cuda")
    rs.route_dup_flags(ctx.h, hd, od, n, max_blocks, fl)
    torch.cuda.synchronize()
    return fl.cpu().numpy()[:n]


@pytest.mark.parametrize("n,max_blocks,seed", [(3000, 512, 1), (5000, 37, 2), (64, 1, 3),
                                               (300, 2048, 4), (2, 2, 5)])
def test_flags_match_direct_check(n, max_blocks, seed):
    offsets, h, want = _case(n, max_blocks, seed)
    got = _run(offsets, h, n, max_blocks)
    assert np.array_equal(got, want)
    if n >= 300:
        assert {0, 1, 2} <= set(got.tolist())


def test_largest_max_blocks():
    # 8192 blocks: one warp's set of 16384 hashes (128 KB of shared memory)
    offsets, h, want = _case(60, 8192, 7, long_frac=0.1, plant_frac=0.5)
    got = _run(offsets, h, 60, 8192)
    assert np.array_equal(got, want)
    assert (want == 1).sum() > 0 and (want == 2).sum() > 0


def test_empty_and_rejected():
    ctx = rs.Context(W=2, K=64)
    h = torch.full((4,), 5, dtype=torch.int64, device="cuda")
    o = torch.zeros(2, dtype=torch.int64, device="cuda")
    f = torch.zeros(1, dtype=torch.uint8, device="cuda")
    rs.route_dup_flags(ctx.h, h, o, 0, 16, f)                  # nothing to do
    for args in ((h, o, 1, 0, f), (h, o, 1, 8193, f), (h, o, -1, 16, f), (None, o, 1, 16, f),
                 (h, None, 1, 16, f), (h, o, 1, 16, None)):
        with pytest.raises(rs.RoutesimError) as e:
            rs.route_dup_flags(ctx.h, *args)
        assert e.value.status == rs.RS_ERR_INVALID
