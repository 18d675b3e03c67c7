"""env_policy_forward_noalloc, the entry point for callers that may not
allocate device memory (a vehicle's control loop with a hard period, or a
host application with a fixed device-memory budget), called through the C
ABI.  Two calls in a row with different weights must equal env_policy_forward
bit for bit (both run the same packing and network kernels), report a clean
status word, leave the device's free memory unchanged after the first
(warm-up) call, and agree with the oracle's bf16 network.  The file is named
so that pytest collects it last."""
import ctypes as C

import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import need_gpu, to_np

pytestmark = pytest.mark.gpu

BF16_TOL = 1e-2     # network outputs against the oracle's bf16 emulation


def _noalloc(lib, pw, vw, obs, head, val, status=None, hidden=256, out=16):
    import torch
    s = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    ptr = lambda t: C.c_void_p(t.data_ptr()) if t is not None else None  # noqa: E731
    return lib.env_policy_forward_noalloc(hidden, out, ptr(pw), ptr(vw), ptr(obs), obs.shape[0],
                                          ptr(head), ptr(val), ptr(status), s)


def test_noalloc_forward_matches_env_policy_forward(oracle):
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    lib = auvenv.lib()
    calls = []
    # every weight region of the shared array changes between the two calls
    for seed, n, bias in ((1, 1000, 0.0), (7, 333, 0.1)):
        w = W.workload("ppo_65536", n_envs=64, weight_seed=seed)
        pw_np, vw_np = W.policy_weights(w, bias), W.value_weights(w, bias)
        obs_np = W.random_observations(10 + seed, n)
        calls.append(dict(
            w=w, pw_np=pw_np, vw_np=vw_np, obs_np=obs_np,
            obs=torch.from_numpy(obs_np).cuda(), pw=torch.from_numpy(pw_np).cuda(),
            vw=torch.from_numpy(vw_np).cuda(),
            head=torch.full((n, 16), float("nan"), device="cuda"),
            val=torch.full((n,), float("nan"), device="cuda"),
            status=torch.full((4,), -7, dtype=torch.int32, device="cuda")))
    torch.cuda.synchronize()
    free = []
    for c in calls:
        free.append(torch.cuda.mem_get_info()[0])
        assert _noalloc(lib, c["pw"], c["vw"], c["obs"], c["head"], c["val"],
                        c["status"]) == auvenv.AUV_OK
        torch.cuda.synchronize()
    free.append(torch.cuda.mem_get_info()[0])
    # after the first (warm-up) call on the device nothing was allocated
    assert free[2] == free[1], (free[1], free[2])
    for k, c in enumerate(calls):
        assert to_np(c["status"]).tolist() == [0, 0, 0, 0], to_np(c["status"])
        env = auvenv.Env(c["w"])
        env.set_weights(c["pw_np"], c["vw_np"])
        n = c["obs"].shape[0]
        head_ref = torch.empty((n, 16), device="cuda")
        val_ref = torch.empty((n,), device="cuda")
        env.policy_forward(c["obs"], head_ref, val_ref)
        torch.cuda.synchronize()
        assert torch.equal(c["head"], head_ref), f"call {k}: head differs"
        assert torch.equal(c["val"], val_ref), f"call {k}: value differs"
        env.close()
    c = calls[1]
    idx = np.r_[0, 1, 100, 332]
    x = c["obs_np"][idx].astype(np.float64)
    eh = np.abs(to_np(c["head"])[idx] - oracle.mlp(c["pw_np"], 18, 256, 16, True, x)).max()
    ev = np.abs(to_np(c["val"])[idx] - oracle.mlp(c["vw_np"], 18, 256, 1, True, x)[:, 0]).max()
    print(f"[no-alloc] against the oracle: head {eh:.3e}, value {ev:.3e} (tol {BF16_TOL})")
    assert eh <= BF16_TOL and ev <= BF16_TOL


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
    st = torch.zeros(5, dtype=torch.int32, device="cuda")
    assert _noalloc(lib, pw, None, x, h, None, status=st.view(torch.uint8)[1:]) == \
        auvenv.AUV_ERR_SIZE
    if torch.cuda.device_count() >= 2:
        # a buffer on another GPU is rejected, not read over the interconnect
        x1 = torch.zeros((4, 18), device="cuda:1")
        assert _noalloc(lib, pw, None, x1, h, None) == auvenv.AUV_ERR_SIZE
