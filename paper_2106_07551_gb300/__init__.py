"""GB300 rollout and payoff-evaluation path of MALib (arXiv 2106.07551).

Thin Python binding over the C ABI of include/malib.h. Names follow the C
entry points (``malib_pop_load``, ``malib_rollout``, ``malib_eval_payoff``);
``Context`` bundles them. Every step of the path runs in the CUDA kernels of
libmalib_gb300.so; this module only marshals arguments (numpy arrays for host
buffers, torch tensors for device buffers) and turns status codes into
exceptions. PyTorch supplies device memory and the CUDA stream.
"""
from __future__ import annotations

import ctypes as C

import numpy as np

from . import _abi
from ._abi import (MALIB_BF16, MALIB_DUMP_LOGITS, MALIB_ENOTCONVERGED, MALIB_ENV_KUHN,
                   MALIB_ENV_LEDUC, MALIB_ENV_SPREAD, MALIB_ENV_ADVERSARY, MALIB_ENV_SPEAKER_LISTENER,
                   MALIB_ENV_PUSH, MALIB_ENV_TAG, MALIB_ENV_REFERENCE, MALIB_EXACT_EXPECTATION, MALIB_F32, MALIB_POL_MLP,
                   MALIB_POL_TABULAR, MALIB_SPREAD_CONTACT, EnvSpec, PolicyDesc, Traj)

__all__ = ["MalibError", "Context", "EnvSpec", "make_spec", "policy_desc", "alloc_traj",
           "alloc_eval_dump", "malib_create", "malib_pop_load", "malib_rollout",
           "malib_eval_payoff", "malib_eval_payoff_ex", "malib_eval_payoff_noalloc", "MALIB_ENV_KUHN", "MALIB_ENV_LEDUC",
           "MALIB_ENV_SPREAD", "MALIB_ENV_ADVERSARY", "MALIB_ENV_SPEAKER_LISTENER", "MALIB_ENV_PUSH",
           "MALIB_ENV_TAG", "MALIB_ENV_REFERENCE", "MALIB_POL_TABULAR", "MALIB_POL_MLP", "MALIB_F32", "MALIB_BF16",
           "MALIB_DUMP_LOGITS", "MALIB_EXACT_EXPECTATION", "MALIB_SPREAD_CONTACT", "MALIB_ENOTCONVERGED"]


class MalibError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{_abi.STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


def _ptr(x):
    """Address of a numpy array or torch tensor (None -> NULL)."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if not x.flags.c_contiguous:
            raise ValueError("arrays passed to the C ABI must be C-contiguous")
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensors passed to the C ABI must be contiguous")
        return x.data_ptr()
    raise TypeError(f"cannot pass {type(x)} to the C ABI")


def make_spec(env_kind, n_agents, obs_dim, n_actions, n_landmarks=0, episode_len=0, n_envs=0,
              flags=0, local_ratio=None) -> EnvSpec:
    """Environment description; local_ratio (spread) weights the reward terms."""
    if local_ratio is not None:
        flags |= _abi.MALIB_SPREAD_LOCAL_RATIO
    return EnvSpec(env_kind, n_agents, n_landmarks, obs_dim, n_actions, episode_len, n_envs,
                   flags, 0.0 if local_ratio is None else float(local_ratio))


def policy_desc(kind, dtype, seat, dims, params) -> PolicyDesc:
    """Descriptor of one population member; params: fp32 numpy array or tensor."""
    d = PolicyDesc()
    d.kind, d.dtype, d.seat = kind, dtype, seat
    d.n_layers = 3 if kind == MALIB_POL_MLP else 1
    for i in range(4):
        d.dims[i] = int(dims[i])
    d.params = _ptr(params)
    d.nbytes = int(params.nbytes if isinstance(params, np.ndarray) else params.numel() * 4)
    return d


def _check(lib, ctx, code):
    if code != 0:
        raise MalibError(code, lib.malib_last_error(ctx).decode(errors="replace"))


def malib_create(device: int = 0, stream=None):
    lib = _abi.load()
    h = C.c_void_p()
    code = lib.malib_create(C.byref(h), device, stream)
    if code != 0:
        raise MalibError(code, lib.malib_last_error(None).decode(errors="replace"))
    return h


def malib_pop_load(ctx, spec: EnvSpec, descs) -> np.ndarray:
    lib = _abi.load()
    arr = (PolicyDesc * len(descs))(*descs)
    ids = np.zeros(len(descs), np.int32)
    _check(lib, ctx, lib.malib_pop_load(ctx, C.byref(spec), arr, len(descs), ids.ctypes.data))
    return ids


def malib_rollout(ctx, spec: EnvSpec, pair_ids, n_episodes: int, seed: int, traj: dict):
    lib = _abi.load()
    n_pairs = int(pair_ids.shape[0])
    t = Traj(_ptr(traj["obs"]), _ptr(traj["action"]), _ptr(traj["reward"]), _ptr(traj["done"]),
             _ptr(traj.get("logits")))
    _check(lib, ctx, lib.malib_rollout(ctx, C.byref(spec), _ptr(pair_ids), n_pairs, n_episodes,
                                       seed, C.byref(t)))


def malib_eval_payoff(ctx, pair_ids, n_episodes: int, seed: int, payoff_out):
    lib = _abi.load()
    _check(lib, ctx, lib.malib_eval_payoff(ctx, _ptr(pair_ids), int(pair_ids.shape[0]),
                                           n_episodes, seed, _ptr(payoff_out)))


def malib_eval_payoff_ex(ctx, pair_ids, n_episodes, seed, flags, payoff_out, dump=None, n_dump=0):
    lib = _abi.load()
    t = None
    if dump is not None:
        t = Traj(_ptr(dump.get("obs")), _ptr(dump.get("action")), _ptr(dump.get("reward")),
                 _ptr(dump.get("done")), _ptr(dump.get("logits")))
    _check(lib, ctx, lib.malib_eval_payoff_ex(ctx, _ptr(pair_ids), int(pair_ids.shape[0]),
                                              n_episodes, seed, flags, _ptr(payoff_out),
                                              C.byref(t) if t is not None else None, n_dump))


def malib_eval_payoff_noalloc(ctx, pair_ids, n_episodes: int, seed: int, payoff_out):
    """Payoff table without any device allocation in the call (device pair table
    and output, at most 8192 pairs); see include/malib.h."""
    lib = _abi.load()
    _check(lib, ctx, lib.malib_eval_payoff_noalloc(ctx, _ptr(pair_ids), int(pair_ids.shape[0]),
                                                   n_episodes, seed, _ptr(payoff_out)))


def alloc_traj(spec: EnvSpec, n_episodes: int, logits: bool = False, device="cuda"):
    """Device trajectory buffers in the layout of include/malib.h."""
    import torch
    E, T, V, N = n_episodes, spec.episode_len, spec.n_envs, spec.n_agents
    P4 = (spec.obs_dim + 3) // 4 * 4
    out = dict(obs=torch.empty((E, T, V, N, P4), dtype=torch.float32, device=device),
               action=torch.empty((E, T, V, N), dtype=torch.uint8, device=device),
               reward=torch.empty((E, T, V, N), dtype=torch.float32, device=device),
               done=torch.empty((E, T, V), dtype=torch.uint8, device=device))
    if logits:
        out["logits"] = torch.empty((E, T, V, N, spec.n_actions), dtype=torch.float32,
                                    device=device)
    return out


def alloc_eval_dump(env_kind: int, n_pairs: int, n_dump: int, device="cuda"):
    """Device dump buffers of malib_eval_payoff_ex (first n_dump hands per pair)."""
    import torch
    S, P4, A = (3, 0, 2) if env_kind == MALIB_ENV_KUHN else (8, 20, 3)
    out = dict(action=torch.empty((n_pairs, n_dump, S), dtype=torch.uint8, device=device),
               reward=torch.empty((n_pairs, n_dump, S), dtype=torch.float32, device=device),
               done=torch.empty((n_pairs, n_dump, S), dtype=torch.uint8, device=device),
               logits=torch.empty((n_pairs, n_dump, S, A), dtype=torch.float32, device=device))
    if P4:
        out["obs"] = torch.empty((n_pairs, n_dump, S, P4), dtype=torch.float32, device=device)
    return out


class Context:
    """One library context on one GPU, ordered on a CUDA stream (default: the
    current torch stream of that device)."""

    def __init__(self, device: int = 0, stream=None):
        self.lib = _abi.load()
        if stream is None:
            import torch
            stream = torch.cuda.current_stream(device).cuda_stream
        elif hasattr(stream, "cuda_stream"):
            stream = stream.cuda_stream
        self.handle = malib_create(device, stream)
        self.device = device

    def close(self):
        if getattr(self, "handle", None):
            self.lib.malib_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def last_error(self) -> str:
        return self.lib.malib_last_error(self.handle).decode(errors="replace")

    def sync(self):
        _check(self.lib, self.handle, self.lib.malib_sync(self.handle))

    def pop_load(self, spec: EnvSpec, descs) -> np.ndarray:
        return malib_pop_load(self.handle, spec, descs)

    def pop_reset(self):
        _check(self.lib, self.handle, self.lib.malib_pop_reset(self.handle))

    def rollout(self, spec, pair_ids, n_episodes, seed, traj):
        malib_rollout(self.handle, spec, pair_ids, n_episodes, seed, traj)

    def eval_payoff(self, pair_ids, n_episodes, seed, payoff_out=None):
        if payoff_out is None:
            payoff_out = np.zeros((int(pair_ids.shape[0]), 4), np.float64)
        malib_eval_payoff(self.handle, pair_ids, n_episodes, seed, payoff_out)
        return payoff_out

    def eval_payoff_ex(self, pair_ids, n_episodes, seed, flags, payoff_out=None, dump=None,
                       n_dump=0):
        if payoff_out is None:
            payoff_out = np.zeros((int(pair_ids.shape[0]), 4), np.float64)
        malib_eval_payoff_ex(self.handle, pair_ids, n_episodes, seed, flags, payoff_out, dump,
                             n_dump)
        return payoff_out

    def eval_decisions(self) -> int:
        """Decisions (env-steps) played by the last Monte-Carlo evaluation."""
        n = C.c_int64(0)
        _check(self.lib, self.handle, self.lib.malib_eval_stats(self.handle, C.byref(n)))
        return int(n.value)

    def launch_count(self) -> int:
        return int(self.lib.malib_launch_count(self.handle))

    def set_timing(self, on: bool):
        _check(self.lib, self.handle, self.lib.malib_set_timing(self.handle, int(on)))

    def main_kernel_ms(self, reset: bool = False):
        n = C.c_int64(0)
        ms = self.lib.malib_main_kernel_ms(self.handle, C.byref(n), int(reset))
        return ms, n.value

    # ---- meta-game solvers (device fp64 tensors; payoff [G][m][n] or [G][m][n][stride]) ----
    @staticmethod
    def _table(payoff, stride):
        G, m, n = int(payoff.shape[0]), int(payoff.shape[1]), int(payoff.shape[2])
        if not payoff.is_contiguous():
            raise ValueError("payoff must be contiguous")
        return G, m, n, int(stride)

    def meta_fictitious_play(self, payoff, iters, x_out, y_out, bounds_out, stride=1):
        """Fictitious play on G games: x_out [G][m], y_out [G][n], bounds_out [G][2]."""
        G, m, n, st = self._table(payoff, stride)
        _check(self.lib, self.handle,
               self.lib.malib_meta_fictitious_play(self.handle, _ptr(payoff), G, m, n, st,
                                                   int(iters), _ptr(x_out), _ptr(y_out),
                                                   _ptr(bounds_out)))

    def meta_lp_nash(self, payoff, x_out, y_out, value_out, stride=1, max_pivots=None):
        """LP equilibrium of G games: x_out [G][m], y_out [G][n], value_out [G].
        max_pivots caps the simplex pivots per game (None: the library's default
        limit); a game over the cap raises ENOTCONVERGED at the next sync()."""
        G, m, n, st = self._table(payoff, stride)
        if max_pivots is None:
            rc = self.lib.malib_meta_lp_nash(self.handle, _ptr(payoff), G, m, n, st, _ptr(x_out),
                                             _ptr(y_out), _ptr(value_out))
        else:
            rc = self.lib.malib_meta_lp_nash_ex(self.handle, _ptr(payoff), G, m, n, st,
                                                int(max_pivots), _ptr(x_out), _ptr(y_out),
                                                _ptr(value_out))
        _check(self.lib, self.handle, rc)

    def meta_aggregate(self, payoff, x, y, row_out, col_out, value_out, stride=1):
        """A y -> row_out [G][m], x^T A -> col_out [G][n], x^T A y -> value_out [G]."""
        G, m, n, st = self._table(payoff, stride)
        _check(self.lib, self.handle,
               self.lib.malib_meta_aggregate(self.handle, _ptr(payoff), G, m, n, st, _ptr(x),
                                             _ptr(y), _ptr(row_out), _ptr(col_out),
                                             _ptr(value_out)))

    def learn_pg(self, spec, pair_ids, n_episodes, traj, policy_id, gamma, entropy_coef, grad_out,
                 stats_out=None):
        """Policy-gradient step of one policy on a rollout's samples: the
        gradient (policy-parameter layout) into grad_out and (M, baseline,
        loss, mean entropy) into stats_out (fp64 [4]); host or device buffers."""
        t = Traj(_ptr(traj["obs"]), _ptr(traj["action"]), _ptr(traj["reward"]), None, None)
        _check(self.lib, self.handle,
               self.lib.malib_learn_pg(self.handle, C.byref(spec), _ptr(pair_ids), int(pair_ids.shape[0]),
                                       n_episodes, C.byref(t), policy_id, gamma, entropy_coef,
                                       _ptr(grad_out), _ptr(stats_out) if stats_out is not None else None))

    def learn_pg_batch(self, spec, pair_ids, n_episodes, traj, policy_ids, gamma, entropy_coef, grad_out,
                       stats_out=None):
        """learn_pg for several distinct policies in one call: grad_out
        [n][P] and stats_out [n][4], host or device."""
        ids = np.ascontiguousarray(policy_ids, np.int32)
        t = Traj(_ptr(traj["obs"]), _ptr(traj["action"]), _ptr(traj["reward"]), None, None)
        _check(self.lib, self.handle,
               self.lib.malib_learn_pg_batch(self.handle, C.byref(spec), _ptr(pair_ids), int(pair_ids.shape[0]),
                                             n_episodes, C.byref(t), _ptr(ids), len(ids), gamma, entropy_coef,
                                             _ptr(grad_out), _ptr(stats_out) if stats_out is not None else None))

    def learn_ppo_batch(self, spec, pair_ids, n_episodes, traj, policy_ids, gamma, entropy_coef, clip_eps,
                        grad_out, stats_out=None):
        """learn_pg_batch with PPO's clipped surrogate against the behavior
        logits traj["logits"] that the rollout recorded (MALIB_DUMP_LOGITS)."""
        ids = np.ascontiguousarray(policy_ids, np.int32)
        lg = traj.get("logits")
        t = Traj(_ptr(traj["obs"]), _ptr(traj["action"]), _ptr(traj["reward"]), None,
                 _ptr(lg) if lg is not None else None)
        _check(self.lib, self.handle,
               self.lib.malib_learn_ppo_batch(self.handle, C.byref(spec), _ptr(pair_ids), int(pair_ids.shape[0]),
                                              n_episodes, C.byref(t), _ptr(ids), len(ids), gamma, entropy_coef,
                                              clip_eps, _ptr(grad_out),
                                              _ptr(stats_out) if stats_out is not None else None))

    def adam_step(self, params, grad, m, v, step, lr, beta1=0.9, beta2=0.999, eps=1e-8):
        """One Adam step on device buffers (parameters, gradient, moments) in place."""
        n = int(params.numel()) if hasattr(params, "numel") else int(params.size)
        _check(self.lib, self.handle,
               self.lib.malib_adam_step(self.handle, _ptr(params), _ptr(grad), _ptr(m), _ptr(v), n, step,
                                        lr, beta1, beta2, eps))

    def pop_update(self, policy_id, params):
        """Replaces a loaded policy's parameters (same shape), host or device."""
        nbytes = int(params.numel()) * 4 if hasattr(params, "numel") else int(params.size) * 4
        _check(self.lib, self.handle, self.lib.malib_pop_update(self.handle, policy_id, _ptr(params), nbytes))

    def exploitability(self, ids0, x, ids1, y):
        """(b0, b1, exploitability) of the seat mixtures (ids with fp64 weights)."""
        ids0 = np.ascontiguousarray(ids0, np.int32)
        ids1 = np.ascontiguousarray(ids1, np.int32)
        x = np.ascontiguousarray(x, np.float64)
        y = np.ascontiguousarray(y, np.float64)
        out = np.zeros(3, np.float64)
        _check(self.lib, self.handle,
               self.lib.malib_exploitability(self.handle, _ptr(ids0), _ptr(x), len(ids0),
                                             _ptr(ids1), _ptr(y), len(ids1), _ptr(out)))
        return float(out[0]), float(out[1]), float(out[2])

    def selftest_philox(self, ctr, seed, out):
        _check(self.lib, self.handle,
               self.lib.malib_selftest_philox(self.handle, _ptr(ctr), seed, _ptr(out),
                                              int(ctr.shape[0])))

    def philox_digest(self, seed, calls, out):
        """out[t] = XOR of the 4 words of Philox calls i < calls at counter
        (t lo, t hi, i, 0) under seed (device uint32 tensor, one entry per t)."""
        _check(self.lib, self.handle,
               self.lib.malib_philox_digest(self.handle, seed, int(out.numel()), int(calls),
                                            _ptr(out)))

    def selftest_wait(self, arrive, limit_ns):
        """A bounded device wait that expires (arrive False) or completes (True);
        the outcome is reported by the next sync()."""
        _check(self.lib, self.handle, self.lib.malib_selftest_wait(self.handle, int(bool(arrive)),
                                                                   int(limit_ns)))

    def selftest_det_expf(self, x, y):
        _check(self.lib, self.handle,
               self.lib.malib_selftest_det_expf(self.handle, _ptr(x), _ptr(y), int(x.numel())))

    def selftest_mma(self, dtype, A, B, D):
        """D = A . B^T on the tensor cores (A [128][K], B [N][K]; bf16 bits or fp32)."""
        N, K = int(B.shape[0]), int(B.shape[1])
        _check(self.lib, self.handle,
               self.lib.malib_selftest_mma(self.handle, dtype, _ptr(A), _ptr(B), _ptr(D), N, K))

    def selftest_mlp_tc(self, policy_id, x, out, reps=1):
        """logits out [n][A] of policy policy_id on rows x [n][in] (device fp32)
        through the pipelined tensor-core engine."""
        _check(self.lib, self.handle,
               self.lib.malib_selftest_mlp_tc(self.handle, int(policy_id), _ptr(x), int(x.shape[0]),
                                              int(reps), _ptr(out)))

    def selftest_sample(self, logits, legal, u, out):
        n, A = logits.shape
        _check(self.lib, self.handle,
               self.lib.malib_selftest_sample(self.handle, _ptr(logits), _ptr(legal), _ptr(u),
                                              A, _ptr(out), n))
