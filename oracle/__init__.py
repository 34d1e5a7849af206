"""CPU oracle for the rollout / payoff-evaluation path (test infrastructure).

A plain, slow CPU restatement of the method (Sec. 3.1 combinations and
rollouts, Sec. 3.2 payoff table, Sec. 4.2 Monte-Carlo evaluation, App. B.1
simple spread) in ``malib_oracle.cpp``, wrapped here with ctypes + numpy.
Only the tests, the smoke check and the benchmark's CPU-baseline leg may use
it; the GPU path never imports it and shares no code with it.

Parity pins live in ``tests/test_oracle_*.py``. The spread episode return under
sampled policies has no closed form: beyond single steps, invariants and two
forced-action episodes (at rest; under a constant force) it is "parity
unpinned".
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "malib_oracle.cpp")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (-O2, no fused multiply-add contraction)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-pthread", _SRC, "-o", tmp]
    subprocess.check_call(cmd)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _L():
    global _lib
    with _lock:
        if _lib is None:
            lib = C.CDLL(build())
            P = C.c_void_p
            i32, i64, u64, f32 = C.c_int32, C.c_int64, C.c_uint64, C.c_float
            sig = {
                "orc_philox": (None, [P, u64, P, i64]),
                "orc_det_expf": (None, [P, P, i64]),
                "orc_det_log1pf": (None, [P, P, i64]),
                "orc_contact_force": (None, [f32, f32, f32, f32, f32, P]),
                "orc_sample": (None, [P, P, P, C.c_int, P, i64]),
                "orc_bf16_round": (f32, [f32]),
                "orc_mlp_forward": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, P, i64, P]),
                "orc_kuhn_exact": (C.c_double, [P, P]),
                "orc_kuhn_eval": (None, [P, P, i32, i64, u64, P, P, i64, C.c_int]),
                "orc_kuhn_hands": (None, [P, P, u64, i64, u64, P]),
                "orc_leduc_deal": (None, [u64, u64, P]),
                "orc_leduc_play": (C.c_int, [C.c_int, C.c_int, C.c_int, P, C.c_int, P, P, P, P, P, P]),
                "orc_leduc_exact": (C.c_double, [P, P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int]),
                "orc_leduc_eval": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, P, i32, i64,
                                          i64, u64, P, i64, P, P, P, P, P, P, P, P, C.c_int]),
                "orc_spread_step": (None, [C.c_int, C.c_int, P, P, P, C.c_float, C.c_int]),
                "orc_spread_obs": (None, [C.c_int, C.c_int, P, C.c_int, P]),
                "orc_spread_reset": (None, [C.c_int, C.c_int, u64, u64, P]),
                "orc_spread_rollout": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int,
                                              C.c_int, C.c_int, C.c_int, i64, i64, i64, P, i32, i64,
                                              u64, P, P, P, P, P, C.c_int, C.c_float, C.c_int]),
                "orc_sl_reset": (None, [u64, u64, P]),
                "orc_sl_step": (None, [P, P, P]),
                "orc_sl_obs": (None, [P, P]),
                "orc_sl_rollout": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, i64, i64, i64,
                                          P, i32, i64, u64, P, P, P, P, P, C.c_int]),
                "orc_adversary_reset": (None, [u64, u64, P]),
                "orc_adversary_step": (None, [P, P, P]),
                "orc_adversary_obs": (None, [P, P]),
                "orc_adversary_rollout": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, i64, i64, i64,
                                                 P, i32, i64, u64, P, P, P, P, P, C.c_int]),
                "orc_push_reset": (None, [u64, u64, P]),
                "orc_push_step": (None, [P, P, P]),
                "orc_push_obs": (None, [P, P]),
                "orc_push_rollout": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, i64, i64, i64,
                                            P, i32, i64, u64, P, P, P, P, P, C.c_int]),
                "orc_ref_reset": (None, [u64, u64, P]),
                "orc_ref_step": (None, [P, P, P, f32]),
                "orc_ref_obs": (None, [P, P]),
                "orc_ref_rollout": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, i64, i64, i64,
                                           P, i32, i64, u64, P, P, P, P, P, C.c_int, f32]),
                "orc_tag_reset": (None, [u64, u64, P]),
                "orc_tag_step": (None, [P, P, P]),
                "orc_tag_obs": (None, [P, P]),
                "orc_tag_rollout": (None, [P, C.c_int, C.c_int, C.c_int, C.c_int, i64, i64, i64,
                                           P, i32, i64, u64, P, P, P, P, P, C.c_int]),
            }
            for name, (res, args) in sig.items():
                fn = getattr(lib, name)
                fn.restype = res
                fn.argtypes = args
            _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


# ---------------------------------------------------------------- primitives
def philox(ctr: np.ndarray, seed: int) -> np.ndarray:
    """Philox4x32-10 of counters uint32 [n][4] under key (seed lo, seed hi)."""
    ctr = _c(ctr, np.uint32).reshape(-1, 4)
    out = np.empty_like(ctr)
    _L().orc_philox(_p(ctr), C.c_uint64(seed), _p(out), ctr.shape[0])
    return out


def det_expf(x: np.ndarray) -> np.ndarray:
    x = _c(x, np.float32)
    y = np.empty_like(x)
    _L().orc_det_expf(_p(x), _p(y), x.size)
    return y


def det_log1pf(x: np.ndarray) -> np.ndarray:
    """log(1 + x) for x in [0, 1] by the fp32 atanh series (contact model)."""
    x = _c(x, np.float32)
    y = np.empty_like(x)
    _L().orc_det_log1pf(_p(x), _p(y), x.size)
    return y


def contact_force(a, b, dmin: float):
    """Soft contact force on the disk at a from the disk at b (radii summing to
    dmin): (force [2] fp32, whether one acts)."""
    out = np.zeros(3, np.float32)
    _L().orc_contact_force(float(a[0]), float(a[1]), float(b[0]), float(b[1]), float(dmin), _p(out))
    return out[:2].copy(), bool(out[2])


def sample(logits: np.ndarray, legal: np.ndarray, u: np.ndarray) -> np.ndarray:
    logits = _c(logits, np.float32)
    n, A = logits.shape
    legal = _c(legal, np.uint8).reshape(n, A)
    u = _c(u, np.float32).reshape(n)
    out = np.empty(n, dtype=np.int32)
    _L().orc_sample(_p(logits), _p(legal), _p(u), A, _p(out), n)
    return out


def bf16_round(x: float) -> float:
    return _L().orc_bf16_round(float(x))


def mlp_forward(params: np.ndarray, dims, x: np.ndarray, bf16: bool = False) -> np.ndarray:
    params = _c(params, np.float32)
    i, h1, h2, o = dims
    x = _c(x, np.float32).reshape(-1, i)
    out = np.empty((x.shape[0], o), dtype=np.float32)
    _L().orc_mlp_forward(_p(params), i, h1, h2, o, int(bf16), _p(x), x.shape[0], _p(out))
    return out


# ---------------------------------------------------------------- Kuhn
def kuhn_exact(pol0: np.ndarray, pol1: np.ndarray) -> float:
    a, b = _c(pol0, np.float32), _c(pol1, np.float32)
    return _L().orc_kuhn_exact(_p(a), _p(b))


def kuhn_eval(tables: np.ndarray, pairs: np.ndarray, n_episodes: int, seed: int,
              n_trace: int = 0, n_threads: int = 0):
    """Monte-Carlo payoff table. Returns (res [n][4], trace int32 [n][n_trace][8] | None)."""
    tables = _c(tables, np.float32).reshape(-1, 6)
    pairs = _c(pairs, np.int32).reshape(-1, 2)
    n = pairs.shape[0]
    res = np.zeros((n, 4), dtype=np.float64)
    trace = np.zeros((n, n_trace, 8), dtype=np.int32) if n_trace else None
    _L().orc_kuhn_eval(_p(tables), _p(pairs), n, n_episodes, C.c_uint64(seed), _p(res),
                       _p(trace), n_trace, n_threads)
    return res, trace


def kuhn_hands(pol0: np.ndarray, pol1: np.ndarray, g0: int, n: int, seed: int) -> np.ndarray:
    """Traces int32 [n][8] (as kuhn_eval's) of the hands with global ids g0 .. g0 + n - 1."""
    a, b = _c(pol0, np.float32), _c(pol1, np.float32)
    trace = np.zeros((n, 8), dtype=np.int32)
    _L().orc_kuhn_hands(_p(a), _p(b), C.c_uint64(g0), n, C.c_uint64(seed), _p(trace))
    return trace


# ---------------------------------------------------------------- Leduc
def leduc_deal(g: int, seed: int):
    out = np.zeros(3, dtype=np.int32)
    _L().orc_leduc_deal(C.c_uint64(g), C.c_uint64(seed), _p(out))
    return tuple(int(v) for v in out)


def leduc_play(c0: int, c1: int, pub: int, actions):
    acts = _c(list(actions), np.int32)
    n = max(1, len(actions))
    payoff = np.zeros(1, np.int32)
    contrib = np.zeros(2, np.int32)
    seats = np.zeros(n, np.int32)
    obs = np.zeros((n, 17), np.float32)
    legal = np.zeros((n, 3), np.uint8)
    done = np.zeros(1, np.int32)
    used = _L().orc_leduc_play(c0, c1, pub, _p(acts), len(actions), _p(payoff), _p(contrib),
                               _p(seats), _p(obs), _p(legal), _p(done))
    return dict(used=used, payoff0=int(payoff[0]), contrib=tuple(int(v) for v in contrib),
                seats=seats[:max(used, 0)], obs=obs[:max(used, 0)], legal=legal[:max(used, 0)],
                done=bool(done[0]))


def leduc_exact(p0: np.ndarray, p1: np.ndarray, dims, bf16: bool = False) -> float:
    a, b = _c(p0, np.float32), _c(p1, np.float32)
    return _L().orc_leduc_exact(_p(a), _p(b), *dims, int(bf16))


def _param_table(params_list):
    arrs = [_c(p, np.float32) for p in params_list]
    tbl = (C.c_void_p * len(arrs))(*[a.ctypes.data for a in arrs])
    return arrs, tbl


def leduc_eval(params_list, dims, pairs, n_episodes, seed, bf16=False, n_rec=0,
               ext_logits=None, n_threads=0, n_sim=None, decisions=None):
    """Monte-Carlo payoff table for Leduc pairs; optional records of the first
    n_rec episodes of every pair (and replay of external logits for them).
    Only hands [0, n_sim) of each pair are simulated (default: all n_episodes);
    episode ids still follow g = pair * n_episodes + e. `decisions`, an int64
    array [n_pairs], receives each pair's number of decisions."""
    n_sim = n_episodes if n_sim is None else n_sim
    arrs, tbl = _param_table(params_list)
    pairs = _c(pairs, np.int32).reshape(-1, 2)
    n = pairs.shape[0]
    res = np.zeros((n, 4), np.float64)
    rec = None
    ptrs = [None] * 6
    if n_rec:
        rec = dict(obs=np.zeros((n, n_rec, 8, 17), np.float32),
                   logits=np.zeros((n, n_rec, 8, 3), np.float32),
                   action=np.full((n, n_rec, 8), -1, np.int8),
                   seat=np.full((n, n_rec, 8), -1, np.int8),
                   payoff=np.zeros((n, n_rec), np.int32),
                   ndec=np.zeros((n, n_rec), np.int32))
        ptrs = [rec[k] for k in ("obs", "logits", "action", "seat", "payoff", "ndec")]
    ext = None if ext_logits is None else _c(ext_logits, np.float32).reshape(n, n_rec, 8, 3)
    _L().orc_leduc_eval(C.cast(tbl, C.c_void_p), *dims, int(bf16), _p(pairs), n, n_episodes,
                        n_sim, C.c_uint64(seed), _p(res), n_rec, _p(ext), *[_p(a) for a in ptrs],
                        _p(decisions), n_threads)
    del arrs
    return res, rec


# ---------------------------------------------------------------- spread
def spread_step(state: np.ndarray, N: int, L: int, actions,
                local_ratio=None, contact: bool = False) -> tuple[np.ndarray, np.ndarray]:
    """One transition; local_ratio (None: the unweighted reward) weights the
    shared cover term by 1 - local_ratio and the agent's collisions by it;
    contact adds the soft contact forces between the agents."""
    st = _c(state, np.float32).copy()
    act = _c(actions, np.int32)
    rew = np.zeros(N, np.float32)
    _L().orc_spread_step(N, L, _p(st), _p(act), _p(rew),
                         -1.0 if local_ratio is None else float(local_ratio), int(bool(contact)))
    return st, rew


def spread_obs(state: np.ndarray, N: int, L: int, obs_dim: int) -> np.ndarray:
    st = _c(state, np.float32)
    out = np.zeros((N, obs_dim), np.float32)
    _L().orc_spread_obs(N, L, _p(st), obs_dim, _p(out))
    return out


def spread_reset(N: int, L: int, g: int, seed: int) -> np.ndarray:
    st = np.zeros(4 * N + 2 * L, np.float32)
    _L().orc_spread_reset(N, L, C.c_uint64(g), C.c_uint64(seed), _p(st))
    return st


def spread_rollout(params_list, dims, N, L, T, n_envs, pairs, n_episodes, seed, bf16=False,
                   env_lo=0, env_hi=None, ext_logits=None, n_threads=0, local_ratio=None,
                   contact=False):
    """Rollout over envs [env_lo, env_hi). Returns dict of obs [E][T][W][N][in],
    action int8 [E][T][W][N], reward [E][T][W][N], logits [E][T][W][N][A]."""
    env_hi = n_envs if env_hi is None else env_hi
    W = env_hi - env_lo
    i, h1, h2, A = dims
    arrs, tbl = _param_table(params_list)
    pairs = _c(pairs, np.int32).reshape(-1, N)
    out = dict(obs=np.zeros((n_episodes, T, W, N, i), np.float32),
               action=np.zeros((n_episodes, T, W, N), np.int8),
               reward=np.zeros((n_episodes, T, W, N), np.float32),
               logits=np.zeros((n_episodes, T, W, N, A), np.float32))
    ext = None if ext_logits is None else _c(ext_logits, np.float32).reshape(n_episodes, T, W, N, A)
    _L().orc_spread_rollout(C.cast(tbl, C.c_void_p), i, h1, h2, A, int(bf16), N, L, T, n_envs,
                            env_lo, env_hi, _p(pairs), pairs.shape[0], n_episodes,
                            C.c_uint64(seed), _p(ext), _p(out["obs"]), _p(out["action"]),
                            _p(out["reward"]), _p(out["logits"]), n_threads,
                            -1.0 if local_ratio is None else float(local_ratio), int(bool(contact)))
    del arrs
    return out


# ---- simple adversary (App. B.1) ----
# state: px,py,vx,vy of agents 0 (adversary), 1, 2; lx,ly of landmarks 0, 1;
# then the target landmark's index (17 floats).
ADV_N, ADV_L, ADV_OBS, ADV_STATE = 3, 2, 14, 17


SL_N, SL_L, SL_OBS, SL_STATE = 2, 3, 11, 16


def sl_reset(g: int, seed: int) -> np.ndarray:
    """Simple speaker listener: state [px,py,vx,vy] x 2, [lx,ly] x 3, target, message."""
    st = np.zeros(SL_STATE, np.float32)
    _L().orc_sl_reset(C.c_uint64(g), C.c_uint64(seed), _p(st))
    return st


def sl_step(state: np.ndarray, actions) -> tuple[np.ndarray, np.ndarray]:
    """One transition; actions [message, move]; rewards [speaker, listener]."""
    st = _c(state, np.float32).copy()
    act = _c(actions, np.int32)
    rew = np.zeros(SL_N, np.float32)
    _L().orc_sl_step(_p(st), _p(act), _p(rew))
    return st, rew


def sl_obs(state: np.ndarray) -> np.ndarray:
    st = _c(state, np.float32)
    out = np.zeros((SL_N, SL_OBS), np.float32)
    _L().orc_sl_obs(_p(st), _p(out))
    return out


def sl_rollout(params_list, dims, T, n_envs, pairs, n_episodes, seed, bf16=False,
               env_lo=0, env_hi=None, ext_logits=None, n_threads=0):
    """Rollout over envs [env_lo, env_hi) of the simple speaker listener (2
    agents, obs 11, 5 actions, the speaker's 3 and 4 illegal). Returns the
    arrays of spread_rollout."""
    env_hi = n_envs if env_hi is None else env_hi
    W = env_hi - env_lo
    i, h1, h2, A = dims
    assert i == SL_OBS and A == 5
    arrs, tbl = _param_table(params_list)
    pairs = _c(pairs, np.int32).reshape(-1, SL_N)
    out = dict(obs=np.zeros((n_episodes, T, W, SL_N, i), np.float32),
               action=np.zeros((n_episodes, T, W, SL_N), np.int8),
               reward=np.zeros((n_episodes, T, W, SL_N), np.float32),
               logits=np.zeros((n_episodes, T, W, SL_N, A), np.float32))
    ext = None if ext_logits is None else _c(ext_logits, np.float32).reshape(n_episodes, T, W, SL_N, A)
    _L().orc_sl_rollout(C.cast(tbl, C.c_void_p), h1, h2, int(bf16), T, n_envs, env_lo, env_hi,
                        _p(pairs), pairs.shape[0], n_episodes, C.c_uint64(seed), _p(ext),
                        _p(out["obs"]), _p(out["action"]), _p(out["reward"]), _p(out["logits"]),
                        n_threads)
    del arrs
    return out


def adversary_reset(g: int, seed: int) -> np.ndarray:
    st = np.zeros(ADV_STATE, np.float32)
    _L().orc_adversary_reset(C.c_uint64(g), C.c_uint64(seed), _p(st))
    return st


def adversary_step(state: np.ndarray, actions) -> tuple[np.ndarray, np.ndarray]:
    """One transition; rewards [adversary, good, good]."""
    st = _c(state, np.float32).copy()
    act = _c(actions, np.int32)
    rew = np.zeros(ADV_N, np.float32)
    _L().orc_adversary_step(_p(st), _p(act), _p(rew))
    return st, rew


def adversary_obs(state: np.ndarray) -> np.ndarray:
    st = _c(state, np.float32)
    out = np.zeros((ADV_N, ADV_OBS), np.float32)
    _L().orc_adversary_obs(_p(st), _p(out))
    return out


def adversary_rollout(params_list, dims, T, n_envs, pairs, n_episodes, seed, bf16=False,
                      env_lo=0, env_hi=None, ext_logits=None, n_threads=0):
    """Rollout over envs [env_lo, env_hi) of the simple adversary (3 agents,
    obs 14, 5 actions). Returns the arrays of spread_rollout."""
    env_hi = n_envs if env_hi is None else env_hi
    W = env_hi - env_lo
    i, h1, h2, A = dims
    assert i == ADV_OBS and A == 5
    arrs, tbl = _param_table(params_list)
    pairs = _c(pairs, np.int32).reshape(-1, ADV_N)
    out = dict(obs=np.zeros((n_episodes, T, W, ADV_N, i), np.float32),
               action=np.zeros((n_episodes, T, W, ADV_N), np.int8),
               reward=np.zeros((n_episodes, T, W, ADV_N), np.float32),
               logits=np.zeros((n_episodes, T, W, ADV_N, A), np.float32))
    ext = None if ext_logits is None else _c(ext_logits, np.float32).reshape(n_episodes, T, W, ADV_N, A)
    _L().orc_adversary_rollout(C.cast(tbl, C.c_void_p), h1, h2, int(bf16), T, n_envs, env_lo,
                               env_hi, _p(pairs), pairs.shape[0], n_episodes, C.c_uint64(seed),
                               _p(ext), _p(out["obs"]), _p(out["action"]), _p(out["reward"]),
                               _p(out["logits"]), n_threads)
    del arrs
    return out


# ---- simple push and simple tag (App. B.1) ----
# push state: px,py,vx,vy of agents 0 (adversary), 1 (good); lx,ly of the
# landmark (10 floats). tag state: px,py,vx,vy of agents 0..2 (adversaries), 3
# (good); ox,oy of the two obstacles (20 floats).
PUSH_N, PUSH_L, PUSH_OBS, PUSH_STATE = 2, 1, 8, 10
TAG_N, TAG_L, TAG_OBS, TAG_STATE = 4, 2, 16, 20


def _scen(name, N, OBS, STATE):
    def reset(g: int, seed: int) -> np.ndarray:
        st = np.zeros(STATE, np.float32)
        getattr(_L(), f"orc_{name}_reset")(C.c_uint64(g), C.c_uint64(seed), _p(st))
        return st

    def step(state: np.ndarray, actions) -> tuple[np.ndarray, np.ndarray]:
        st = _c(state, np.float32).copy()
        act = _c(actions, np.int32)
        rew = np.zeros(N, np.float32)
        getattr(_L(), f"orc_{name}_step")(_p(st), _p(act), _p(rew))
        return st, rew

    def obs(state: np.ndarray) -> np.ndarray:
        st = _c(state, np.float32)
        out = np.zeros((N, OBS), np.float32)
        getattr(_L(), f"orc_{name}_obs")(_p(st), _p(out))
        return out

    def rollout(params_list, dims, T, n_envs, pairs, n_episodes, seed, bf16=False,
                env_lo=0, env_hi=None, ext_logits=None, n_threads=0):
        env_hi = n_envs if env_hi is None else env_hi
        W = env_hi - env_lo
        i, h1, h2, A = dims
        assert i == OBS and A == 5
        arrs, tbl = _param_table(params_list)
        prs = _c(pairs, np.int32).reshape(-1, N)
        out = dict(obs=np.zeros((n_episodes, T, W, N, i), np.float32),
                   action=np.zeros((n_episodes, T, W, N), np.int8),
                   reward=np.zeros((n_episodes, T, W, N), np.float32),
                   logits=np.zeros((n_episodes, T, W, N, A), np.float32))
        ext = None if ext_logits is None else _c(ext_logits, np.float32).reshape(n_episodes, T, W, N, A)
        getattr(_L(), f"orc_{name}_rollout")(
            C.cast(tbl, C.c_void_p), h1, h2, int(bf16), T, n_envs, env_lo, env_hi, _p(prs),
            prs.shape[0], n_episodes, C.c_uint64(seed), _p(ext), _p(out["obs"]),
            _p(out["action"]), _p(out["reward"]), _p(out["logits"]), n_threads)
        del arrs
        return out

    return reset, step, obs, rollout


push_reset, push_step, push_obs, push_rollout = _scen("push", PUSH_N, PUSH_OBS, PUSH_STATE)
push_rollout.__doc__ = """Rollout over envs [env_lo, env_hi) of the simple push (2 agents, obs 8,
5 actions). Returns the arrays of spread_rollout."""
tag_reset, tag_step, tag_obs, tag_rollout = _scen("tag", TAG_N, TAG_OBS, TAG_STATE)
tag_rollout.__doc__ = """Rollout over envs [env_lo, env_hi) of the simple tag (4 agents, obs 16,
5 actions). Returns the arrays of spread_rollout."""


# ---- simple reference (App. B.1) ----
# state: px,py,vx,vy of agents 0, 1; lx,ly of the three landmarks; the two goals;
# the two last messages (-1: none) (18 floats). Action a = 5 * message + move.
REF_N, REF_L, REF_OBS, REF_A, REF_STATE = 2, 3, 14, 15, 18


def ref_reset(g: int, seed: int) -> np.ndarray:
    st = np.zeros(REF_STATE, np.float32)
    _L().orc_ref_reset(C.c_uint64(g), C.c_uint64(seed), _p(st))
    return st


def ref_step(state: np.ndarray, actions, local_ratio: float = 0.5) -> tuple[np.ndarray, np.ndarray]:
    st = _c(state, np.float32).copy()
    act = _c(actions, np.int32)
    rew = np.zeros(REF_N, np.float32)
    _L().orc_ref_step(_p(st), _p(act), _p(rew), float(local_ratio))
    return st, rew


def ref_obs(state: np.ndarray) -> np.ndarray:
    st = _c(state, np.float32)
    out = np.zeros((REF_N, REF_OBS), np.float32)
    _L().orc_ref_obs(_p(st), _p(out))
    return out


def ref_rollout(params_list, dims, T, n_envs, pairs, n_episodes, seed, bf16=False,
                env_lo=0, env_hi=None, ext_logits=None, n_threads=0, local_ratio=None):
    """Rollout over envs [env_lo, env_hi) of the simple reference (2 agents,
    obs 14, 15 actions); local_ratio None: 0.5. Returns the arrays of
    spread_rollout."""
    env_hi = n_envs if env_hi is None else env_hi
    W = env_hi - env_lo
    i, h1, h2, A = dims
    assert i == REF_OBS and A == REF_A
    arrs, tbl = _param_table(params_list)
    prs = _c(pairs, np.int32).reshape(-1, REF_N)
    out = dict(obs=np.zeros((n_episodes, T, W, REF_N, i), np.float32),
               action=np.zeros((n_episodes, T, W, REF_N), np.int8),
               reward=np.zeros((n_episodes, T, W, REF_N), np.float32),
               logits=np.zeros((n_episodes, T, W, REF_N, A), np.float32))
    ext = None if ext_logits is None else _c(ext_logits, np.float32).reshape(n_episodes, T, W, REF_N, A)
    _L().orc_ref_rollout(C.cast(tbl, C.c_void_p), h1, h2, int(bf16), T, n_envs, env_lo, env_hi, _p(prs),
                         prs.shape[0], n_episodes, C.c_uint64(seed), _p(ext), _p(out["obs"]),
                         _p(out["action"]), _p(out["reward"]), _p(out["logits"]), n_threads,
                         0.5 if local_ratio is None else float(local_ratio))
    del arrs
    return out
