"""The synthetic layer-set shapes reproduce the paper's trainable-parameter counts
(Table 3): RoI learns one logit per weight (M per group), the categorical
parameterisation C(M, N) per group."""
import json
import math
import os

import pytest

import workloads as W

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "table3_trainable_params.json")))


@pytest.mark.parametrize("name", list(W.LAYER_SETS))
def test_roi_parameter_counts(name):
    billions = W.LAYER_SETS[name].elements / 1e9
    assert abs(billions - GOLD["roi_billions"][name]) <= GOLD["printed_resolution_billions"]


def test_categorical_ratio():
    for nm, ratio in GOLD["maskllm_ratio"].items():
        N, M = map(int, nm.split(":"))
        assert math.comb(M, N) / M == ratio
    for name, roi in GOLD["roi_billions"].items():
        assert abs(GOLD["maskllm_billions_2of4"][name] - 1.5 * roi) <= 0.051
        assert abs(GOLD["maskllm_billions_2of8"][name] - 3.5 * roi) <= 0.051


def test_set_sizes():
    assert W.LAYER_SETS["qwen2.5-7b"].elements == 6_525_288_448
    assert W.LAYER_SETS["qwen2.5-0.5b"].elements == 357_826_560
    for cfg in W.CONFIGS.values():
        for N, M in cfg.nm:
            if cfg.layer_set:
                for _, _, r, c in W.LAYER_SETS[cfg.layer_set].tensors():
                    assert c % M == 0 and (r * c) % 32 == 0
