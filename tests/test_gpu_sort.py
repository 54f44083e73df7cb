"""The library's stable radix sort (akashic_mem_sort_pairs) against numpy's
stable argsort: both the small form (at most 256 tiles of 1024 pairs: one
launch a pass, offsets and next-pass histograms built by the scatter) and
the large form (tiles of 4096 pairs: tile histograms, a scan, a scatter per
pass), at ragged sizes on both sides of the switch and of a small tile,
with narrow and full key widths and many equal keys (stability)."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

TILE = 4096
SMALL_TILE = 1024
SMALL_MAX = 256 * SMALL_TILE


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05708_gb300 import _build
    _build.build()


def _check(n, bits, key_hi, seed):
    import torch
    from paper_2607_05708_gb300 import sort_pairs
    rng = np.random.default_rng(seed)
    keys = rng.integers(0, key_hi, size=n, dtype=np.uint64).astype(np.uint32)
    vals = np.arange(n, dtype=np.uint32) * np.uint32(2654435761)   # distinct, unordered
    mask = np.uint32(0xffffffff) if bits == 32 else np.uint32((1 << bits) - 1)
    order = np.argsort(keys & mask, kind="stable")
    kd = torch.from_numpy(keys.view(np.int32)).cuda()
    vd = torch.from_numpy(vals.view(np.int32)).cuda()
    sort_pairs(kd, vd, bits)
    got_k = kd.cpu().numpy().view(np.uint32)
    got_v = vd.cpu().numpy().view(np.uint32)
    np.testing.assert_array_equal(got_k, keys[order])
    np.testing.assert_array_equal(got_v, vals[order])


@pytest.mark.parametrize("n", [2, 31, SMALL_TILE - 1, SMALL_TILE, SMALL_TILE + 1, TILE - 1, TILE,
                               TILE + 1, 32 * TILE, 131_071,
                               SMALL_MAX - 1, SMALL_MAX, SMALL_MAX + 1, 1_000_003])
@pytest.mark.parametrize("bits", [5, 8, 20, 32])
def test_sort_pairs_matches_stable_argsort(n, bits):
    # keys drawn from a range about n / 8 wide: many equal keys in every case
    _check(n, bits, key_hi=max(2, n // 8) if bits < 32 else 1 << 32, seed=n * 41 + bits)


def test_sort_pairs_low_bits_only_and_trivial_cases():
    # only the low bits order the pairs: the high bits travel along untouched
    _check(50_000, 12, key_hi=1 << 32, seed=7)
    _check(50_000, 0, key_hi=1 << 32, seed=8)      # bits = 0: nothing moves
    _check(1, 32, key_hi=1 << 32, seed=9)
