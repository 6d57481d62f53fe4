"""The analytic cost / storage model against the numbers the paper prints (Sec. 3.5, Table 'cost')."""
import json
import os

import pytest

from paper_2608_23794_gb300 import costmodel as cm

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_cost_numbers.json")))


def _round(v, digits):
    return round(v, digits)


def test_resnet50_replaced_macs():
    ps = cm.resnet_entrance_projections(cm.RESNET_BLOCKS["resnet50"])
    assert len(ps) == GOLD["resnet50_replaced_projections"]["value"]
    dense = sum(cm.dense_macs(p) for p in ps) / 1e6
    moce = sum(cm.moce_macs(p, 8) for p in ps) / 1e6
    gate = sum(cm.gate_macs(p, 8) for p in ps) / 1e9
    assert _round(dense, 1) == GOLD["resnet50_replaced_dense_macs_M"]["value"]
    assert _round(moce, 1) == GOLD["resnet50_replaced_moce_macs_M"]["value"]
    assert round(dense / moce) == GOLD["resnet50_replaced_reduction_x"]["value"]
    assert _round(gate, 5) == GOLD["resnet50_gate_macs_G"]["value"]


def test_resnet50_storage():
    ps = cm.resnet_entrance_projections(cm.RESNET_BLOCKS["resnet50"])
    weights = sum(p.C * p.E for p in ps) / 1e6
    logits = sum(cm.deployed_logits(p, 8) for p in ps) / 1e3
    idx_kb = sum(cm.index_bytes(p, 8) for p in ps) / 1e3
    assert _round(weights, 2) == GOLD["resnet50_replaced_weights_M"]["value"]
    assert _round(logits, 1) == GOLD["resnet50_retained_logits_k"]["value"]
    assert round(idx_kb) == GOLD["resnet50_index_bytes_KB"]["value"]


@pytest.mark.parametrize("row", GOLD["break_even"])
def test_break_even(row):
    assert round(cm.break_even_k(row["C"], row["E"])) == row["k_star"]


@pytest.mark.parametrize("net", ["resnet50", "resnet101", "resnet152"])
def test_network_macs_and_params(net):
    # network MACs: dense total minus the replaced dense projections plus their MoCE cost
    blocks = cm.RESNET_BLOCKS[net]
    ps = cm.resnet_entrance_projections(blocks)
    g = GOLD["network_macs_G"][net]
    moce_total = g["dense"] - sum(cm.dense_macs(p) for p in ps) / 1e9 + \
        sum(cm.moce_macs(p, 8) for p in ps) / 1e9
    assert _round(moce_total, 3) == g["moce"]
    prm = cm.moce_network_params(blocks, k=8)
    gp = GOLD["params_M"][net]
    assert _round(prm["dense"] / 1e6, 2) == gp["dense"]
    assert _round(prm["train"] / 1e6, 2) == gp["moce_train"]
    assert _round(prm["deploy"] / 1e6, 2) == gp["moce_deploy"]


def test_arithmetic_intensity():
    ai = GOLD["arithmetic_intensity_flop_per_byte"]
    pr = ai["projection"]
    got = cm.arithmetic_intensity(cm.Projection(pr["C"], pr["E"], pr["H"], pr["W"]), ai["k"],
                                  ai["batch"], ai["bytes_per_element"])
    assert round(got["dense"]) == ai["dense"]
    assert round(got["moce"], 1) == ai["moce"]


def test_ratio_bound_holds():
    for p in cm.resnet_entrance_projections():
        r = cm.moce_macs(p, 8) / cm.dense_macs(p)
        assert r <= cm.ratio_bound(p.C, p.E, 8) + 1e-12
