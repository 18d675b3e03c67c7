"""The C-ABI library builds, loads, exports every entry point that
include/auvenv.h declares, and rejects bad configurations before touching
the GPU (no compute calls here)."""
import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "auvenv.h")


@pytest.fixture(scope="module")
def auvlib():
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    return auvenv.lib()


def header_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\**\s*((?:env|ppo|rbuf|auv_probe)_\w+|auv_gemm\w*)\s*\(", text,
                                 flags=re.M)))


def test_header_declares_the_entry_points():
    names = header_functions()
    for must in ("env_create", "env_reset", "env_step", "env_rollout", "env_step_actions",
                 "env_gae", "ppo_create", "ppo_grads", "ppo_apply", "ppo_update"):
        assert must in names


def test_library_exports_every_declared_symbol(auvlib):
    from paper_2512_13359_gb300 import auvenv
    names = header_functions()
    assert sorted(auvenv.EXPORTED) == names
    out = subprocess.run(["nm", "-D", "--defined-only", auvenv.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT\s+(\w+)$", out, flags=re.M))
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        assert hasattr(auvlib, n)
    assert auvlib.env_abi_version() == 3


def test_config_struct_size_matches_header(auvlib):
    """sizeof(auv_config) as compiled equals the binding's mirror: a create
    with the binding's size passes the version guard, any other size fails."""
    from paper_2512_13359_gb300 import auvenv, workloads as W
    cfg = auvenv.make_config(W.workload("tiny_64"))
    h = C.c_void_p()
    cfg.struct_size = C.sizeof(auvenv.AuvConfig) + 4
    rc = auvlib.env_create(C.byref(cfg), None, C.byref(h))
    assert rc == auvenv.AUV_ERR_INVALID
    assert b"struct_size" in auvlib.env_last_error(None)


@pytest.mark.parametrize("field,value,code", [
    ("n_envs", 0, -1), ("substeps", 0, -1), ("substeps", 65, -1), ("episode_len", 0, -1),
    ("dt", 0.0, -1), ("dt", float("nan"), -1), ("mass", -1.0, -1), ("policy_out", 12, -1),
    ("mlp_mode", 7, -1), ("goal_yaw_range", 4.0, -1), ("hidden", 128, -6),
])
def test_invalid_configs_are_rejected(auvlib, field, value, code):
    from paper_2512_13359_gb300 import auvenv, workloads as W
    cfg = auvenv.make_config(W.workload("tiny_64"))
    setattr(cfg, field, value)
    h = C.c_void_p()
    rc = auvlib.env_create(C.byref(cfg), None, C.byref(h))
    assert rc == code, auvlib.env_last_error(None)
    assert not h.value


@pytest.mark.parametrize("field,value,code", [
    ("model", 5, -1), ("mavg_len", 0, -1), ("mavg_len", 9, -1), ("policy_out", 8, -1),
    ("goal_att_range", 4.0, -1), ("fluid_density", -1.0, -1), ("f_max", float("inf"), -1),
    ("hidden", 128, -6),
])
def test_invalid_paper_model_configs_are_rejected(auvlib, field, value, code):
    from paper_2512_13359_gb300 import auvenv, workloads as W
    cfg = auvenv.make_config(W.workload("paper_tiny"))
    setattr(cfg, field, value)
    h = C.c_void_p()
    rc = auvlib.env_create(C.byref(cfg), None, C.byref(h))
    assert rc == code, auvlib.env_last_error(None)
    assert not h.value


def test_paper_model_needs_an_inertia_box(auvlib):
    """The inertia fluid model needs a box with the body's moments: each
    principal moment below the sum of the other two."""
    from paper_2512_13359_gb300 import auvenv, workloads as W
    cfg = auvenv.make_config(W.workload("paper_tiny", inertia=(0.5, 0.1, 0.1)))
    h = C.c_void_p()
    assert auvlib.env_create(C.byref(cfg), None, C.byref(h)) == auvenv.AUV_ERR_INVALID
    assert b"inertia box" in auvlib.env_last_error(None)


def test_layout_of_each_model(auvlib):
    from paper_2512_13359_gb300 import auvenv, workloads as W
    f = auvenv.layout(auvenv.AUV_MODEL_FOSSEN)
    assert (f.obs_dim, f.act_dim, f.state_fields, f.param_fields) == (
        W.OBS_DIM, W.ACT_DIM, W.STATE_FIELDS, W.PARAM_FIELDS)
    p = auvenv.layout(auvenv.AUV_MODEL_PAPER)
    assert (p.obs_dim, p.act_dim, p.state_fields, p.param_fields) == (
        W.PAPER_OBS_DIM, W.PAPER_ACT_DIM, W.PAPER_STATE_FIELDS, W.PAPER_PARAM_FIELDS)
    out = auvenv.AuvLayout()
    assert auvlib.env_layout(7, C.byref(out)) == auvenv.AUV_ERR_INVALID
    assert auvlib.env_layout(0, None) == auvenv.AUV_ERR_INVALID


def test_bf16_mode_requires_the_built_shape(auvlib):
    from paper_2512_13359_gb300 import auvenv, workloads as W
    cfg = auvenv.make_config(W.workload("ppo_65536", hidden=64))
    h = C.c_void_p()
    assert auvlib.env_create(C.byref(cfg), None, C.byref(h)) == auvenv.AUV_ERR_UNSUPPORTED


def test_null_arguments(auvlib):
    from paper_2512_13359_gb300 import auvenv
    h = C.c_void_p()
    assert auvlib.env_create(None, None, C.byref(h)) == auvenv.AUV_ERR_INVALID
    assert auvlib.env_destroy(None) == auvenv.AUV_ERR_INVALID
    assert auvlib.env_reset(None, None, None) == auvenv.AUV_ERR_INVALID
    assert auvlib.env_rollout(None, 1, None, None) == auvenv.AUV_ERR_INVALID


def test_ppo_config_struct_size_matches_header(auvlib):
    from paper_2512_13359_gb300 import auvenv
    cfg = auvenv.make_ppo_config(18, 8, 256, 4096)
    h = C.c_void_p()
    cfg.struct_size = C.sizeof(auvenv.PpoConfig) - 4
    assert auvlib.ppo_create(C.byref(cfg), C.byref(h)) == auvenv.AUV_ERR_INVALID
    assert b"struct_size" in auvlib.ppo_last_error(None)


@pytest.mark.parametrize("field,value,msg", [
    ("obs_dim", 0, b"obs_dim"), ("obs_dim", 65, b"obs_dim"), ("act_dim", 9, b"act_dim"),
    ("hidden", 100, b"hidden"), ("hidden", 2048, b"hidden"), ("minibatch", 1, b"minibatch"),
    ("precision", 3, b"precision"), ("norm_adv", 2, b"norm_adv"), ("flags", 4, b"flags"),
    ("clip_eps", 0.0, b"clip_eps"), ("clip_eps", float("nan"), b"clip_eps"),
    ("vf_coef", float("inf"), b"finite"), ("max_grad_norm", float("nan"), b"finite"),
    ("lr", -1e-3, b"lr"), ("adam_beta1", 1.0, b"betas"), ("adam_beta2", -0.1, b"betas"),
    ("adam_eps", 0.0, b"adam_eps"), ("logstd_min", 3.0, b"logstd")])
def test_invalid_ppo_configs_are_rejected(auvlib, field, value, msg):
    from paper_2512_13359_gb300 import auvenv
    cfg = auvenv.make_ppo_config(18, 8, 256, 4096)
    setattr(cfg, field, value)
    h = C.c_void_p()
    assert auvlib.ppo_create(C.byref(cfg), C.byref(h)) == auvenv.AUV_ERR_INVALID
    assert msg in auvlib.ppo_last_error(None)
    assert not h.value


def test_ppo_null_arguments(auvlib):
    from paper_2512_13359_gb300 import auvenv
    h = C.c_void_p()
    E = auvenv.AUV_ERR_INVALID
    assert auvlib.ppo_create(None, C.byref(h)) == E
    assert auvlib.ppo_destroy(None) == E
    assert auvlib.ppo_grads(None, None, 0, 0, None, None, None) == E
    assert auvlib.ppo_apply(None, None, None, None) == E
    assert auvlib.ppo_update(None, None, 1, 1, None, None) == E
    assert auvlib.ppo_set_weights(None, None, None, None) == E


def test_binding_fails_loudly_without_the_library(tmp_path):
    from paper_2512_13359_gb300 import auvenv
    saved = auvenv._lib
    auvenv._lib = None
    try:
        with pytest.raises(auvenv.LibraryMissing):
            auvenv.lib(str(tmp_path / "missing.so"))
    finally:
        auvenv._lib = saved
