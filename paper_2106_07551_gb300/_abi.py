"""ctypes declarations of the C ABI in include/malib.h (argument marshalling only).

Loading fails loudly when libmalib_gb300.so has not been built: there is no
CPU fallback for any entry point.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

from . import build as _build

MALIB_OK, MALIB_EINVAL, MALIB_ENOMEM, MALIB_ECUDA = 0, -1, -2, -3
MALIB_ESTATE, MALIB_ETIMEOUT, MALIB_EUNSUPPORTED = -4, -5, -6
MALIB_ENOTCONVERGED = -7
STATUS_NAMES = {0: "OK", -1: "EINVAL", -2: "ENOMEM", -3: "ECUDA", -4: "ESTATE", -5: "ETIMEOUT",
                -6: "EUNSUPPORTED", -7: "ENOTCONVERGED"}

MALIB_ENV_KUHN, MALIB_ENV_LEDUC, MALIB_ENV_SPREAD, MALIB_ENV_ADVERSARY = 1, 2, 3, 4
MALIB_ENV_SPEAKER_LISTENER, MALIB_ENV_PUSH, MALIB_ENV_TAG, MALIB_ENV_REFERENCE = 5, 6, 7, 8
MALIB_POL_TABULAR, MALIB_POL_MLP = 1, 2
MALIB_F32, MALIB_BF16 = 0, 1
MALIB_DUMP_LOGITS, MALIB_EXACT_EXPECTATION, MALIB_SPREAD_LOCAL_RATIO = 1, 2, 4
MALIB_SPREAD_CONTACT = 8

# Every symbol include/malib.h declares.
EXPORTS = (
    "malib_create", "malib_destroy", "malib_last_error", "malib_sync", "malib_set_stream",
    "malib_pop_load", "malib_pop_reset", "malib_rollout", "malib_eval_payoff",
    "malib_eval_payoff_ex", "malib_eval_payoff_noalloc", "malib_eval_stats", "malib_launch_count",
    "malib_set_timing", "malib_main_kernel_ms",
    "malib_selftest_philox", "malib_philox_digest", "malib_selftest_wait", "malib_selftest_det_expf",
    "malib_selftest_sample",
    "malib_selftest_mma", "malib_selftest_mlp_tc", "malib_meta_fictitious_play", "malib_meta_lp_nash",
    "malib_meta_lp_nash_ex",
    "malib_meta_aggregate", "malib_exploitability", "malib_learn_pg", "malib_learn_pg_batch",
    "malib_learn_ppo_batch", "malib_adam_step",
    "malib_pop_update",
)


class EnvSpec(C.Structure):
    _fields_ = [("env_kind", C.c_int32), ("n_agents", C.c_int32), ("n_landmarks", C.c_int32),
                ("obs_dim", C.c_int32), ("n_actions", C.c_int32), ("episode_len", C.c_int32),
                ("n_envs", C.c_int64), ("flags", C.c_uint32), ("local_ratio", C.c_float)]


class PolicyDesc(C.Structure):
    _fields_ = [("kind", C.c_int32), ("dtype", C.c_int32), ("seat", C.c_int32),
                ("n_layers", C.c_int32), ("dims", C.c_int32 * 4), ("params", C.c_void_p),
                ("nbytes", C.c_int64)]


class Traj(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("action", C.c_void_p), ("reward", C.c_void_p),
                ("done", C.c_void_p), ("logits", C.c_void_p)]


_lock = threading.Lock()
_lib = None


def lib_path() -> str:
    return _build.LIB_PATH


def load(path: str | None = None):
    """Loads libmalib_gb300.so (built by build.build()); raises if it is missing."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = path or lib_path()
        if not os.path.exists(path):
            raise ImportError(
                f"{path} is missing: build the CUDA library first "
                "(python -c 'import __graft_entry__ as g; g.build()'); there is no CPU fallback")
        L = C.CDLL(path)
        P, i32, i64, u32, u64 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint32, C.c_uint64
        sig = {
            "malib_create": (C.c_int, [C.POINTER(P), C.c_int, P]),
            "malib_destroy": (None, [P]),
            "malib_last_error": (C.c_char_p, [P]),
            "malib_sync": (C.c_int, [P]),
            "malib_set_stream": (C.c_int, [P, P]),
            "malib_pop_load": (C.c_int, [P, C.POINTER(EnvSpec), C.POINTER(PolicyDesc), i32, P]),
            "malib_pop_reset": (C.c_int, [P]),
            "malib_rollout": (C.c_int, [P, C.POINTER(EnvSpec), P, i32, i64, u64, C.POINTER(Traj)]),
            "malib_eval_payoff": (C.c_int, [P, P, i32, i64, u64, P]),
            "malib_eval_payoff_ex": (C.c_int, [P, P, i32, i64, u64, u32, P, C.POINTER(Traj), i64]),
            "malib_eval_payoff_noalloc": (C.c_int, [P, P, i32, i64, u64, P]),
            "malib_eval_stats": (C.c_int, [P, C.POINTER(C.c_int64)]),
            "malib_launch_count": (C.c_int64, [P]),
            "malib_set_timing": (C.c_int, [P, C.c_int]),
            "malib_main_kernel_ms": (C.c_double, [P, C.POINTER(C.c_int64), C.c_int]),
            "malib_selftest_philox": (C.c_int, [P, P, u64, P, i64]),
            "malib_philox_digest": (C.c_int, [P, u64, i64, i32, P]),
            "malib_selftest_wait": (C.c_int, [P, i32, i64]),
            "malib_selftest_det_expf": (C.c_int, [P, P, P, i64]),
            "malib_selftest_sample": (C.c_int, [P, P, P, P, i32, P, i64]),
            "malib_selftest_mma": (C.c_int, [P, i32, P, P, P, i32, i32]),
            "malib_selftest_mlp_tc": (C.c_int, [P, i32, P, i64, i32, P]),
            "malib_meta_fictitious_play": (C.c_int, [P, P, i32, i32, i32, i32, i64, P, P, P]),
            "malib_meta_lp_nash": (C.c_int, [P, P, i32, i32, i32, i32, P, P, P]),
            "malib_meta_lp_nash_ex": (C.c_int, [P, P, i32, i32, i32, i32, i32, P, P, P]),
            "malib_meta_aggregate": (C.c_int, [P, P, i32, i32, i32, i32, P, P, P, P, P]),
            "malib_exploitability": (C.c_int, [P, P, P, i32, P, P, i32, P]),
            "malib_learn_pg": (C.c_int, [P, C.POINTER(EnvSpec), P, i32, i64, C.POINTER(Traj), i32, C.c_float,
                                         C.c_float, P, P]),
            "malib_learn_pg_batch": (C.c_int, [P, C.POINTER(EnvSpec), P, i32, i64, C.POINTER(Traj), P, i32,
                                               C.c_float, C.c_float, P, P]),
            "malib_learn_ppo_batch": (C.c_int, [P, C.POINTER(EnvSpec), P, i32, i64, C.POINTER(Traj), P, i32,
                                                C.c_float, C.c_float, C.c_float, P, P]),
            "malib_adam_step": (C.c_int, [P, P, P, P, P, i64, i64, C.c_float, C.c_float, C.c_float, C.c_float]),
            "malib_pop_update": (C.c_int, [P, i32, P, i64]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
        return _lib
