"""Helpers shared by the GPU parity tests: build the library and an Env for a
workload, seed the oracle with the same env ids, and the tolerance metric
|gpu - oracle| <= rtol * max(|oracle|, floor) (floors: 1 m, 1 for the
quaternion, 1 m/s, 1 rad/s; every state row has floor 1)."""
import numpy as np
import pytest

STATE_TOL = 1e-5        # per-step state, fp32 path vs double oracle
REWARD_SUM_TOL = 1e-4   # accumulated reward over 100 steps, relative


def need_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_13359_gb300 import build
    build.build()
    return torch


def make_env(w, policy=True, bias_std=0.0):
    from paper_2512_13359_gb300 import auvenv, workloads as W
    env = auvenv.Env(w)
    if policy:
        pw = W.policy_weights(w, bias_std)
        vw = W.value_weights(w, bias_std) if w["has_value"] else None
        env.set_weights(pw, vw)
    return env


def oracle_batch(oracle, m, ids):
    b = oracle.Batch(np.asarray(ids))
    oracle.reset(m, b)
    return b


def rel_err(gpu, ref, floor=1.0):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return np.abs(gpu - ref) / np.maximum(np.abs(ref), floor)


def assert_close(gpu, ref, tol, floor=1.0, what=""):
    e = rel_err(gpu, ref, floor)
    if e.size and not np.all(e <= tol):
        idx = np.unravel_index(np.argmax(e), e.shape)
        raise AssertionError(f"{what}: max rel err {e.max():.3e} > {tol:.1e} at {idx}: "
                             f"gpu {np.asarray(gpu)[idx]!r} oracle {np.asarray(ref)[idx]!r}")


def to_np(t):
    return t.detach().cpu().numpy()


def u32(t):
    return to_np(t).view(np.uint32)
