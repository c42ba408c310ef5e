"""Host-side input generators: shapes, determinism, the Zipf law."""
import numpy as np
import pytest

from paper_2609_37899_gb300 import inputs


@pytest.mark.parametrize("name", list(inputs.CONFIGS))
def test_config_shapes_and_determinism(name):
    c = inputs.CONFIGS[name]
    b = inputs.config_batch(name, batch=min(c["batch"], 4))
    assert b.dtype == np.uint8
    assert b.shape == (c["n_experts"], min(c["batch"], 4), c["seq_len"] + 1)
    assert (inputs.config_batch(name, batch=min(c["batch"], 4)) == b).all()
    assert (inputs.config_batch(name, step=1, batch=min(c["batch"], 4)) != b).any()


def test_param_counts():
    assert inputs.param_count(32, 64) == 49_664
    assert inputs.param_count(64, 960) == 4_198_400
    assert inputs.param_count(64, 1376) == 8_300_160
    assert inputs.param_count(64, 480) == 1_185_920
    assert inputs.param_count(32, 48) == 36_288
    o = inputs.param_offsets(64, 960)
    assert o["end"] == inputs.param_count(64, 960)


def test_zipf_conditionals():
    x = inputs.expert_batch(1, 512, 512, 1, 0, 0)[0]
    cnt = np.zeros((256, 256))
    np.add.at(cnt, (x[:, :-1].ravel(), x[:, 1:].ravel()), 1)
    rows = cnt[cnt.sum(1) > 600]
    top = -np.sort(-rows / rows.sum(1, keepdims=True), axis=1)
    p = np.diff(np.r_[0.0, inputs.zipf_cdf(1.1)])
    assert top[:, 0].mean() == pytest.approx(p[0], abs=0.01)
    assert top[:, 1].mean() == pytest.approx(p[1], abs=0.01)


def test_clusters_differ_and_mixture():
    b = inputs.expert_batch(2, 64, 64, 1, 0, 0)
    assert (b[0] != b[1]).mean() > 0.9
    m = inputs.expert_batch(1, 64, 64, 2, 0, 0, mixture=(0, 1))
    assert m.shape == (1, 64, 65)


def test_init_params():
    th = inputs.init_params(2, 64, 960, 0)
    o = inputs.param_offsets(64, 960)
    assert th.dtype == np.float32
    assert (th[:, o["b"]:o["w_out"]] == 0).all()
    assert th[:, o["w_hh"]:o["b"]].std() == pytest.approx(1 / np.sqrt(1024), rel=0.01)
    t2 = inputs.init_params(1, 32, 64, 0, std=0.1)
    assert t2.std() == pytest.approx(0.1, rel=0.02)
