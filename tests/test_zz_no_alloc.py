"""env_policy_forward_noalloc, the entry point for callers that may not
allocate device memory (a vehicle's control loop with a hard period, or a
host application with a fixed device-memory budget), called through the C
ABI and checked against env_policy_forward on two calls in a row.  The file
is named so that pytest collects it last."""
import ctypes as C

import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu

TOL = 3e-2      # the bf16 network tolerance of the other tensor-core tests


def _noalloc(lib, pw, vw, obs, head, val, hidden=256, out=16):
    import torch
    s = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    return lib.env_policy_forward_noalloc(hidden, out, C.c_void_p(pw.data_ptr()),
                                          C.c_void_p(vw.data_ptr()) if vw is not None else None,
                                          C.c_void_p(obs.data_ptr()), obs.shape[0],
                                          C.c_void_p(head.data_ptr()),
                                          C.c_void_p(val.data_ptr()) if val is not None else None, s)


def test_noalloc_forward_matches_env_policy_forward():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    lib = auvenv.lib()
    w = W.workload("ppo_65536", n_envs=64)
    for call, (seed, n) in enumerate(((1, 1000), (2, 333))):
        pw_np, vw_np = W.policy_weights(w, 0.1 * call), W.value_weights(w, 0.1 * call)
        obs_np = W.random_observations(10 + seed, n)
        obs = torch.from_numpy(obs_np).cuda()
        pw = torch.from_numpy(pw_np).cuda()
        vw = torch.from_numpy(vw_np).cuda()
        head = torch.full((n, 16), float("nan"), device="cuda")
        val = torch.full((n,), float("nan"), device="cuda")
        assert _noalloc(lib, pw, vw, obs, head, val) == auvenv.AUV_OK
        w_call = dict(w, weight_seed=w["weight_seed"])
        env = auvenv.Env(w_call)
        env.set_weights(pw_np, vw_np)
        head_ref = torch.empty((n, 16), device="cuda")
        val_ref = torch.empty((n,), device="cuda")
        env.policy_forward(obs, head_ref, val_ref)
        torch.cuda.synchronize()
        eh = np.abs(to_np(head) - to_np(head_ref)).max()
        ev = np.abs(to_np(val) - to_np(val_ref)).max()
        print(f"[no-alloc] call {call}: head diff {eh:.3e}, value diff {ev:.3e} (tol {TOL})")
        assert eh <= TOL and ev <= TOL
        env.close()


def test_noalloc_rejects_bad_shapes():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    lib = auvenv.lib()
    x = torch.zeros((4, 18), device="cuda")
    h = torch.zeros((4, 16), device="cuda")
    pw = torch.zeros(W.mlp_param_count(18, 256, 16), device="cuda")
    assert _noalloc(lib, pw, None, x, h, None, hidden=512) == auvenv.AUV_ERR_SIZE
    assert _noalloc(lib, pw, None, x, h, None, out=32) == auvenv.AUV_ERR_SIZE
    assert _noalloc(lib, pw, None, x, h, None, hidden=64) == auvenv.AUV_ERR_UNSUPPORTED
    assert _noalloc(lib, pw, None, x.cpu(), h, None) == auvenv.AUV_ERR_SIZE
