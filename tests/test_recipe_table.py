"""The per-matrix recipe table of the LLaVA-shaped benchmark (a JSON file in
the package): the recipes config 5 names, read the same way by bench.py and by
the binding, each one a recipe the library builds for its shape."""
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TABLE = os.path.join(ROOT, "paper_2505_07531_gb300", "recipes", "llava_v1_6_7b.json")


@pytest.fixture(scope="module")
def qx():
    from paper_2505_07531_gb300 import build

    if not os.path.exists(build.LIB):
        build.build_library()
    import paper_2505_07531_gb300.qx as qx

    return qx


def test_table_holds_the_config_5_recipes(qx):
    t = qx.recipe_table(TABLE)
    lang = {nm: (n, k, r.bits, r.group_size, r.kind) for nm, n, k, r in t["language"]["matrices"]}
    # attention Q/K 3-bit LUT g128; V/O and the MLP 4-bit uniform g64; Llama-7B shapes
    assert lang == {"q_proj": (4096, 4096, 3, 128, 1), "k_proj": (4096, 4096, 3, 128, 1),
                    "v_proj": (4096, 4096, 4, 64, 0), "o_proj": (4096, 4096, 4, 64, 0),
                    "gate_proj": (11008, 4096, 4, 64, 0), "up_proj": (11008, 4096, 4, 64, 0),
                    "down_proj": (4096, 11008, 4, 64, 0)}
    assert t["language"]["layers"] == 32 and t["vision"]["layers"] == 24
    vis = {nm: (n, k, r.bits, r.group_size, r.kind) for nm, n, k, r in t["vision"]["matrices"]}
    assert vis == {"q_proj": (1024, 1024, 4, 128, 0), "k_proj": (1024, 1024, 4, 128, 0),
                   "v_proj": (1024, 1024, 4, 128, 0), "o_proj": (1024, 1024, 4, 128, 0),
                   "fc1": (4096, 1024, 4, 128, 0), "fc2": (1024, 4096, 4, 128, 0)}


def test_bench_and_binding_read_it_alike(qx):
    import sys

    sys.path.insert(0, ROOT)
    import bench

    t = qx.recipe_table(TABLE)
    assert [(nm, n, k, (r.bits, r.group_size, r.kind)) for nm, n, k, r in t["language"]["matrices"]] == \
        [(nm, n, k, rec) for nm, n, k, _, _, rec in bench.LLAVA_LANG]
    assert [(nm, n, k) for nm, n, k, _ in t["vision"]["matrices"]] == [(nm, n, k) for nm, n, k, *_ in bench.LLAVA_VISION]
    assert {(r.bits, r.group_size, r.kind) for *_, r in t["vision"]["matrices"]} == {bench.LLAVA_VISION_RECIPE}


def test_every_recipe_is_built_for_its_shape(qx):
    for sub in qx.recipe_table(TABLE).values():
        for _, n, k, r in sub["matrices"]:
            assert sum(qx.packed_size(n, k, r).values()) > 0
