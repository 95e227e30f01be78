"""The roofline's FLOP counting reproduces the paper's printed App. G numbers."""
import json
import os

import pytest

from paper_2609_08443_gb300 import roofline as rf

G = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "flop_model.json")))
HP = rf.PAPER_HPARAMS
L = 100_000


def _near(x, ref_prec):
    ref, prec = ref_prec
    assert abs(x - ref) <= prec / 2 + 1e-12, (x, ref)


def test_no_mrlb():
    stca = rf.stca_flops(L, HP["n_stca"], HP["D"], HP["h"]) / 1e9
    seq = rf.seqo1_expected_flops(L, 0.5, HP["Ls"], HP["d"], HP["D"], HP["h"], HP["n_sa"],
                                  HP["n_stca"]) / 1e9
    _near(stca, G["no_mrlb"]["stca"])
    _near(seq, G["no_mrlb"]["seqo1"])
    _near(stca / seq, G["no_mrlb"]["ratio"])


@pytest.mark.parametrize("key,R,p", [("train_mrlb", 40, 0.5), ("infer_mrlb", 300, 0.6)])
def test_mrlb(key, R, p):
    stca = rf.stca_mrlb_flops(L, R, HP["n_stca"], HP["D"], HP["h"]) / 1e9
    seq = rf.seqo1_mrlb_expected_flops(L, R, p, HP["Ls"], HP["d"], HP["D"], HP["h"],
                                       HP["n_sa"], HP["n_stca"]) / 1e9
    _near(stca, G[key]["stca"])
    _near(seq, G[key]["seqo1"])
    _near(stca / seq, G[key]["ratio"])
    fig = G["fig1_headline"]["train" if key == "train_mrlb" else "infer"]
    _near(stca / seq, fig)


def test_sketch_step_counts_the_papers_score_and_aggregation_terms():
    # one head, one user: the forward counts exactly the 4 L_s L d of App. G.3
    w = rf.fwd_work(L, 1, 1, HP["Ls"], HP["d"], 2)
    layer_L_terms = rf.sa_layer_flops(L, HP["Ls"], HP["d"]) - rf.sa_layer_flops(0, HP["Ls"], HP["d"])
    assert w.flops == 4 * HP["Ls"] * L * HP["d"]
    assert layer_L_terms - 2 * L * HP["d"] ** 2 == w.flops


def test_roofline_picks_the_slowest_bound():
    w = rf.step_work(12_800_000, 128, 8, 512, 128, 2)
    t = rf.roofline_time(w, 1931.7, 6775.6)
    assert t["bound"] == "tensor"
    assert abs(w.flops - 12 * 512 * 128 * 12_800_000 * 8) < 1
