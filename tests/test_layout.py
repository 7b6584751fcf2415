"""CE-MoE layout tools (composition rule, Sec. 4.1; Algorithm 1, Sec. 4.2)
against the worked outputs the paper prints, plus properties every pattern
must have.  Host-only calls into the library; no GPU needed."""
import os
import shutil

import pytest

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="nvcc is needed to build the library")

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "ce_moe_layout_examples.txt")


@pytest.fixture(scope="module")
def L():
    from paper_2608_28511_gb300 import _build, abi
    _build.build()
    return abi


def _cases(kind):
    out = []
    for line in open(GOLDEN):
        line = line.split("#", 1)[0].strip()
        if line.startswith(kind + " "):
            lhs, rhs = line[len(kind) + 1:].split("->")
            out.append((lhs.split(), rhs.split()))
    return out


@pytest.mark.parametrize("lhs,rhs", _cases("composition"))
def test_composition_matches_the_paper(L, lhs, rhs):
    a_star, b_star, c_star, alpha = int(lhs[0]), int(lhs[1]), int(lhs[2]), float(lhs[3])
    assert L.moe_ce_composition(a_star, b_star, c_star, alpha) == tuple(int(v) for v in rhs)


@pytest.mark.parametrize("lhs,rhs", _cases("pattern"))
def test_layer_pattern_matches_the_paper(L, lhs, rhs):
    pattern, blocks, decorated = L.moe_ce_layer_pattern(*map(int, lhs))
    assert blocks == rhs[0]
    assert decorated == rhs[1]
    assert pattern == rhs[1].replace("[", "").replace("]", "").replace("(", "").replace(")", "")


@pytest.mark.parametrize("lhs,rhs", _cases("composition"))
def test_patterns_of_the_table2_compositions_are_well_formed(L, lhs, rhs):
    a, b, c, d = map(int, rhs)
    pattern, blocks, decorated = L.moe_ce_layer_pattern(a, b, c, d)
    # exactly the composition's blocks, starting with token mixing
    assert (pattern.count("M"), pattern.count("E"), pattern.count("*"), pattern.count("-")) == (a, b, c, d)
    assert pattern[0] == "M"
    # one virtual block per bracket group; attention only in A blocks
    assert len(blocks) == decorated.count("[") + decorated.count("(")
    assert all(("*" in grp) == (k == "A") for k, grp in zip(blocks, decorated.replace("]", "|").replace(")", "|")
                                                               .replace("[", "").replace("(", "").split("|")))


def test_routed_layer_count_and_eq1_volume(L):
    # Sec. 4.1: 23 -> 8 routed layers is 8q instead of 23q all-to-all calls
    a, b, c, d = L.moe_ce_composition(23, 23, 6, 4.0)
    assert round(100 * (1 - b / 23), 1) == 65.2
    shp = L.MoeShape.of(8192, 1, 6, 2688, 128, 1856, "bf16")
    # Eq. 1 scales with L_E: the layer library's per-layer term times the routed layer count
    assert b * L.moe_eq1_bytes(shp) / (23 * L.moe_eq1_bytes(shp)) == pytest.approx(8 / 23)


def test_invalid_compositions_are_rejected(L):
    with pytest.raises(L.MoeError):
        L.moe_ce_layer_pattern(10, 2, 3, 2)      # b < c
    with pytest.raises(L.MoeError):
        L.moe_ce_composition(0, 0, 9, 4.0)       # no room for the attention blocks' partners
