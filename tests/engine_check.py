"""Every-step check of a tensor-core (bf16) rollout against the oracle.

The fused rollout kernel computes, per env and control step, the
observation, the bf16 policy network, the Gaussian draw, the physics
substeps, the reward and the done flag, and writes all of them to the
trajectory.  This module checks every step of such a trajectory for a set of
sampled envs:

- physics: the oracle replays the kernel's own actions act[t] from the same
  reset draw (action replay, so the comparison does not depend on the bf16
  network's rounding): obs[t] of the oracle's state against the kernel's at
  the fp32 tolerance, rew[t] per step, dones bit-exact, reward sums over
  100-step windows, and the final state and counters.  Over a long launch
  the fp32 trajectory drifts from the double one by accumulated rounding
  (about 1e-5 relative after some 400 steps of the paper model); for such
  launches the caller passes the kernel's own state at window starts
  (`resync`, from the same rollout run in windows, which is bit-identical),
  and the oracle restarts from it, so each window is held to the fp32
  tolerance from a common state;
- network and draw: at every t the oracle's bf16 network on the kernel's
  own obs[t], the oracle's log-std clamp and the oracle's normals of global
  step t_g0 + t give a and log pi (oracle.policy_act), and the oracle's
  bf16 value network gives V; the kernel's act, logp and value must agree
  within the bf16 tolerance.

Tolerances.  bf16 network outputs carry at most BF16_TOL (1e-2) absolute
error (measured about 2e-3).  a = mu + sigma eps inherits the error of mu
and sigma eps times that of the log-std, so |da| <= BF16_TOL (1 + sigma
|eps|), with sigma |eps| = |a - mu| taken from the oracle.  log pi sums the
log-std of every action component: |dlogp| <= act_dim * BF16_TOL.  The
kernel's normals use the hardware log and sine (absolute error about 1e-6),
far inside these bounds.

Test infrastructure: used by tests/ and __graft_entry__.smoke() only.
"""
import numpy as np

from paper_2512_13359_gb300 import workloads as W

STATE_TOL = 1e-5          # per-step state and observation, fp32 vs double
REWARD_TOL = 1e-4         # per-step reward (floor 1), and 100-step sums
BF16_TOL = 1e-2           # bf16 network outputs (absolute)


def _rel(gpu, ref, floor=1.0):
    return np.abs(np.asarray(gpu, np.float64) - ref) / np.maximum(np.abs(ref), floor)


def _check(cond, msg):
    if not cond:
        raise AssertionError(msg)


def sample_ids(n, k=40, seed=5):
    """k or more env ids of [0, n): both ends, the first tile boundary and
    random ids."""
    fixed = [0, 1, 127, 128, n - 2, n - 1]
    rnd = np.random.default_rng(seed).integers(0, n, k)
    ids = np.unique(np.clip(np.r_[fixed, rnd], 0, n - 1))
    return ids.astype(np.int64)


def check_engine_rollout(oracle, w, traj, ids, T, t_g0=0, final_state=None, resync=None,
                         net_tol=BF16_TOL):
    """Check the trajectory `traj` (dict of torch tensors or numpy arrays
    with the env's [T][K][N] layout) of a rollout of workload `w` that
    started from the first reset draw at global step t_g0.  final_state:
    optional (state, params, t_ep, episode) arrays of the env after the
    rollout.  resync: optional {t: (state, params, t_ep, episode)} of the
    kernel's batch before step t; the oracle continues from it.  net_tol:
    bound on the network outputs' absolute error (the oracle evaluates the
    workload's network arithmetic: bf16 emulation for bf16 networks, exact
    otherwise).  Returns the measured maxima."""
    paper = W.is_paper(w)
    n_all = int(w["n_envs"])
    ids = np.asarray(ids, dtype=np.int64)
    k = len(ids)
    d, na = W.obs_dim(w), W.act_dim(w)

    def take(key):
        v = traj[key]
        if hasattr(v, "detach"):
            import torch
            return v.detach().index_select(-1, torch.as_tensor(ids, device=v.device)).cpu().numpy()
        return np.asarray(v)[..., ids]

    g = {key: take(key) for key in traj}
    _check(g["obs"].shape == (T, d, k), f"obs shape {g['obs'].shape}")
    m = oracle.paper_model(w) if paper else oracle.model(w)
    b = oracle.PaperBatch(ids) if paper else oracle.Batch(ids)
    (oracle.paper_reset if paper else oracle.reset)(m, b)
    pw = W.policy_weights(w)
    vw = W.value_weights(w) if w["has_value"] else None
    act_fn = oracle.paper_policy_act if paper else oracle.policy_act
    replay = oracle.paper_replay if paper else oracle.replay
    H = int(w["hidden"])
    worst = dict(obs=0.0, rew=0.0, act=0.0, logp=0.0, value=0.0)
    rew_ref = np.zeros((T, k))
    obs_hist = []
    for t in range(T):
        if resync and t in resync:
            st, pr, t_ep, ep = (np.asarray(x) for x in resync[t])
            b.state[:] = st[:, ids]
            b.params[:] = pr[:, ids]
            b.t_ep[:] = t_ep[ids]
            b.episode[:] = ep.view(np.uint32)[ids]
        if paper:
            ref_obs = np.stack([oracle.paper_observe(b.state[:, j], b.params[:, j])
                                for j in range(k)], axis=1)
        else:
            ref_obs = np.stack([oracle.observe(b.state[:, j], b.params[:, j])[0]
                                for j in range(k)], axis=1)
        e = _rel(g["obs"][t], ref_obs)
        worst["obs"] = max(worst["obs"], e.max())
        if e.max() > STATE_TOL:
            kk, jj = np.unravel_index(np.argmax(e), e.shape)
            hist = [float(np.max(_rel(g["obs"][u][:, jj], obs_hist[u][:, jj])))
                    for u in range(max(0, t - 8), t)]
            _check(False, f"obs[{t}]: rel err {e.max():.3e} at component {kk}, env {ids[jj]}: "
                          f"gpu {g['obs'][t][kk, jj]!r} oracle {ref_obs[kk, jj]!r}; env "
                          f"obs errors of the 8 previous steps {hist}; t_ep {b.t_ep[jj]}")
        obs_hist.append(ref_obs)
        o = g["obs"][t].T.astype(np.float64)
        a_ref, lp_ref, mu = act_fn(m, pw, ids.astype(np.uint32), t_g0 + t, o, with_mu=True)
        da = np.abs(g["act"][t].T - a_ref)
        bound = net_tol * (1.0 + np.abs(a_ref - mu))
        worst["act"] = max(worst["act"], (da / (1.0 + np.abs(a_ref - mu))).max())
        _check(np.all(da <= bound), f"act[{t}]: max excess {(da - bound).max():.3e}")
        dl = np.abs(g["logp"][t] - lp_ref)
        worst["logp"] = max(worst["logp"], dl.max())
        _check(dl.max() <= na * net_tol, f"logp[{t}]: {dl.max():.3e}")
        if vw is not None and "value" in g:
            v_ref = oracle.mlp(vw, d, H, 1, True, o)[:, 0]
            dv = np.abs(g["value"][t] - v_ref).max()
            worst["value"] = max(worst["value"], dv)
            _check(dv <= net_tol, f"value[{t}]: {dv:.3e}")
        a_t = np.ascontiguousarray(g["act"][t:t + 1], dtype=np.float32)
        r, dn, _ = replay(m, b, a_t)
        _check(np.array_equal(g["done"][t], dn[0]), f"done[{t}] differs")
        e = _rel(g["rew"][t], r[0])
        worst["rew"] = max(worst["rew"], e.max())
        _check(e.max() <= REWARD_TOL, f"rew[{t}]: rel err {e.max():.3e}")
        rew_ref[t] = r[0]
    for t0 in range(0, T, 100):
        s_g = g["rew"][t0:t0 + 100].astype(np.float64).sum(axis=0)
        s_r = rew_ref[t0:t0 + 100].sum(axis=0)
        e = _rel(s_g, s_r)
        _check(e.max() <= REWARD_TOL, f"reward sum from step {t0}: rel err {e.max():.3e}")
    if final_state is not None:
        st, pr, t_ep, ep = final_state
        e = _rel(np.asarray(st)[:, ids], b.state)
        worst["state"] = e.max()
        _check(e.max() <= STATE_TOL, f"final state: rel err {e.max():.3e}")
        _check(np.array_equal(np.asarray(pr)[:, ids].astype(np.float32),
                              b.params.astype(np.float32)), "final params differ")
        _check(np.array_equal(np.asarray(t_ep)[ids], b.t_ep), "t_ep differs")
        _check(np.array_equal(np.asarray(ep).view(np.uint32)[ids], b.episode), "episode differs")
    _check(n_all >= int(ids.max()) + 1, "sampled id out of range")
    return worst
