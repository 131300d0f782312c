"""The arithmetic the paper prints in its worked example (Appendix B) and introduction."""
import itertools
import json
import math
from pathlib import Path

from oracle import rift_oracle as O
from synth import workloads as W

G = json.loads((Path(__file__).parent / "golden" / "walkthrough_appendix_b.json").read_text())


def test_grid_and_reduction():
    assert G["grid"][0] * G["grid"][1] == G["N"] == 64
    assert math.floor(G["scene_px"][0] / G["tile_px"]) == 8 and math.floor(G["scene_px"][1] / G["tile_px"]) == 8
    assert round(100 * (1 - G["kept"] / G["N"])) == G["vlm_call_reduction_pct"]


def test_paper_constants_are_the_policy_defaults():
    assert sorted(G["budgets_C"]) == list(W.RIFT_POLICY.C)
    assert G["tau"] == W.RIFT_POLICY.tau
    assert G["knn_m"] == W.RIFT400.knn_m
    assert G["tokens_per_tile"] == W.RIFT400.scene.n_v


def test_average_budget_is_reachable_with_the_stated_assignment():
    # 7 object tiles at 72 tokens; the other 10 retained tiles take budgets >= 288 from C.
    # Some such assignment averages 36% (rounded) of the full 576 over the 17 calls.
    C = [c for c in G["budgets_C"] if c >= G["clutter_tile_budget"]]
    n_other = G["kept"] - G["positive_tiles"]
    ok = False
    for combo in itertools.combinations_with_replacement(C, n_other):
        tot = G["positive_tiles"] * G["object_tile_budget"] + sum(combo)
        if round(100 * tot / (G["kept"] * G["tokens_per_tile"])) == G["avg_budget_pct"]:
            ok = True
            break
    assert ok


def test_policy_reproduces_the_inverted_assignment():
    assert O.budget(1.0, W.RIFT_POLICY) == G["object_tile_budget"]
    assert O.budget(0.4, W.RIFT_POLICY) == G["clutter_tile_budget"]


def test_token_counts_of_the_introduction():
    assert round(G["tiles_6700px"] * G["tokens_per_tile"] / 1000) == int(G["vision_tokens_400_tiles"][:-1])
    assert round(G["tiles_fig1"] * G["tokens_per_tile"] / 1000) == int(G["vision_tokens_270_tiles"][:-1])
    assert math.ceil(6700 / G["tile_px"]) ** 2 == G["tiles_6700px"]
    assert W.RIFT400.scene.N == G["tiles_6700px"]
