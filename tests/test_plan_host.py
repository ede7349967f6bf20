"""CPU checks of the tensor-core search planner (oprag_plan_search, no GPU):
every plan fits in a CTA's shared memory, the list slots it provisions cover
every (query tile, CTA) pair that an independent replay of the unit schedule
produces, and the launch modes are the ones the planner documents (dual mode
for small batches, CTA pairs for large batches with buffered lists)."""
import itertools

import pytest

from paper_2608_08340_gb300 import _lib
from paper_2608_08340_gb300 import build as lib_build
from paper_2608_08340_gb300.index import plan_search

MAX_SMEM_PER_CTA = 232448          # 227 KB, the opt-in limit of one CTA


@pytest.fixture(scope="module", autouse=True)
def _built():
    lib_build.build()
    _lib.load()


def list_len(k):
    return 8 if k <= 8 else 16 if k <= 16 else 32 if k <= 32 else 128 if k <= 128 else 256


def first_cta(j, uqt, c):
    return max(0, j * c // uqt - 1)


def replay_slots(p):
    """(schedule query tile, CTA slot) pairs of the unit schedule: corpus
    windows of `win` tiles, units of a window ordered tile-major and cut into
    one contiguous share per slot (a CTA, or a pair of CTAs)."""
    c = p["grid"] // p["cluster"]
    pairs = set()
    w = 0
    while w * p["win"] < p["nt"]:
        tw = min(p["win"], p["nt"] - w * p["win"])
        uw = p["uqt"] * tw
        for cta in range(c):
            lo, hi = uw * cta // c, uw * (cta + 1) // c
            for j in range(lo // tw, (hi - 1) // tw + 1) if lo < hi else ():
                pairs.add((j, cta))
        w += 1
    return pairs, c


SHAPES = list(itertools.product((1000, 4097, 32768, 1 << 20), (64, 768),
                                (1, 32, 129, 256, 300, 512, 2048, 4096), (5, 16, 33, 100),
                                (0, 2, 3)))


@pytest.mark.parametrize("n,d,q,k,force", SHAPES)
def test_plan_fits_and_provisions_every_list(n, d, q, k, force):
    p = plan_search(n, d, q, k, num_sms=148, force_pair=force, pair_capacity=74)
    assert p["smem"] <= MAX_SMEM_PER_CTA
    assert p["grid"] >= 1 and p["grid"] % p["cluster"] == 0
    assert p["qt"] == (q + 127) // 128
    two_tiles = p["dual"] == 1 or p["cluster"] == 2
    assert p["uqt"] == ((p["qt"] + 1) // 2 if two_tiles else p["qt"])
    assert p["nt"] == (n + p["block_n"] - 1) // p["block_n"]
    if p["dual"]:
        assert p["block_n"] == 128 and p["cluster"] == 1 and list_len(k) <= 16
    if p["cluster"] == 2:
        assert p["block_n"] == 256
    # Lists per CTA and query tile: one per epilogue set (two for lists of
    # 8-16 and for buffered lists, one for lists of 32), one in dual mode.
    kl = list_len(k)
    assert p["sets"] == (1 if p["dual"] else (2 if kl <= 16 or kl > 32 else 1))
    # Every (query tile, slot) the schedule produces owns a list slot.
    pairs, c = replay_slots(p)
    per_tile = p["pmax"] // p["sets"]
    for j, cta in pairs:
        pc = cta - first_cta(j, p["uqt"], c)
        assert 0 <= pc < per_tile, (j, cta, p)
    # The scratch holds every list slot.
    kl = list_len(k)
    stride = 2 * kl if kl > 32 else kl
    rows = p["uqt"] * (2 if two_tiles else 1) * p["pmax"] * 128
    assert p["scratch"] >= rows * stride * 8


def test_plan_modes_follow_the_documented_rules():
    # Paper-shaped small batches: dual mode up to four units per CTA.
    for q in (129, 256, 384, 512):
        assert plan_search(32768, 768, q, 5)["dual"] == 1, q
    assert plan_search(32768, 768, 1024, 5)["dual"] == 0
    # One query tile, or lists longer than 16 keys: no dual mode.
    assert plan_search(32768, 768, 128, 5)["dual"] == 0
    assert plan_search(32768, 768, 256, 20)["dual"] == 0
    # Large batches with buffered lists run as CTA pairs, if the device fits them.
    assert plan_search(1 << 20, 768, 2048, 100)["cluster"] == 2
    assert plan_search(1 << 20, 768, 2048, 100, pair_capacity=0)["cluster"] == 1
    assert plan_search(1 << 20, 768, 512, 100)["cluster"] == 1       # 4 query tiles
    assert plan_search(32768, 1024, 4096, 10)["cluster"] == 1        # lists of 16
    # Forced modes: single CTAs never pair; dual needs two tiles and k <= 16.
    assert plan_search(1 << 20, 768, 2048, 100, force_pair=1)["cluster"] == 1
    assert plan_search(32768, 768, 256, 5, force_pair=1)["dual"] == 0
    assert plan_search(32768, 768, 1024, 5, force_pair=3)["dual"] == 1
    assert plan_search(32768, 768, 100, 5, force_pair=3)["dual"] == 0


@pytest.mark.parametrize("args", [
    (0, 768, 1, 5), (100, 0, 1, 5), (100, 768, 0, 5), (100, 768, 1, 0),
    (100, 770, 1, 5), (100, 768, 1, 100000)])
def test_plan_rejects_bad_shapes(args):
    with pytest.raises(_lib.OpragError):
        plan_search(*args)
