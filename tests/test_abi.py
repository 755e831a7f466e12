"""The C-ABI library builds for sm_103a, loads, and exports every symbol that
include/*.h declares (CPU only: no compute call is made)."""
import ctypes
import glob
import os
import re

from harness import ROOT


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^\s*[A-Za-z_][\w\s\*]*?\b(leap_\w+)\s*\(", src, flags=re.M):
            names.add(m.group(1))
    return names


def test_header_declares_the_boundary():
    names = _declared()
    for fn in ("leap_group_rank_advantages", "leap_rollout_token_counts", "leap_scatter_turn_advantages",
               "leap_token_logprobs", "leap_grpo_loss_fwd", "leap_grpo_loss_bwd", "leap_get_device_status"):
        assert fn in names


def test_library_exports_every_declared_symbol():
    from paper_2608_01804_gb300 import build
    path = build.build()
    lib = ctypes.CDLL(path)
    for name in sorted(_declared()):
        assert hasattr(lib, name), name
    from paper_2608_01804_gb300 import leap as L
    assert set(L.EXPORTS) == _declared()
    lib.leap_version.restype = ctypes.c_int32
    assert lib.leap_version() >= 100
    lib.leap_status_string.restype = ctypes.c_char_p
    assert lib.leap_status_string(1) == b"LEAP_ERR_INVALID_ARG"


def test_host_argument_checks_need_no_gpu():
    """Invalid arguments are rejected on the host before any CUDA call."""
    from paper_2608_01804_gb300 import leap as L
    lib = L.lib()
    p = L.RankParams(1, 1, 2, 0, 1, 0.9, 1e-6, 0, 0, 1, 0, 0.5)       # G = 1: Eq. 6 divides by G - 1
    assert lib.leap_group_rank_advantages(ctypes.byref(p), *([None] * 14), None) == L.LEAP_ERR_INVALID_ARG
    p = L.RankParams(1, 8, 9, 0, 1, 0.9, 1e-6, 0, 0, 1, 0, 0.5)       # M > 8
    assert lib.leap_group_rank_advantages(ctypes.byref(p), *([None] * 14), None) == L.LEAP_ERR_INVALID_ARG
    p = L.RankParams(1, 8, 2, 5, 3, 0.9, 1e-6, 0, 0, 1, 0, 0.5)       # tau_min > tau_max
    assert lib.leap_group_rank_advantages(ctypes.byref(p), *([None] * 14), None) == L.LEAP_ERR_INVALID_ARG
    p = L.RankParams(1, 8, 2, 0, 8, 1.5, 1e-6, 0, 0, 1, 0, 0.5)       # gamma > 1
    assert lib.leap_group_rank_advantages(ctypes.byref(p), *([None] * 14), None) == L.LEAP_ERR_INVALID_ARG
    p = L.RankParams(1, 8, 2, 0, 8, 0.9, 1e-6, 0, 0, 1, 0, 1.5)       # static_c > 1
    assert lib.leap_group_rank_advantages(ctypes.byref(p), *([None] * 14), None) == L.LEAP_ERR_INVALID_ARG
    p = L.RankParams(1, 8, 2, 0, 8, 0.9, 1e-6, 1, 0, 1, 0, 0.5)       # LEXI without speedup / tokens
    pt = ctypes.c_void_p(256)
    assert lib.leap_group_rank_advantages(ctypes.byref(p), pt, pt, None, None, None, None, None, None, None,
                                          None, None, pt, pt, None, None) == L.LEAP_ERR_INVALID_ARG
    # ld not a multiple of 8 / misaligned logits.
    assert lib.leap_token_logprobs(ctypes.c_void_p(16), 1001, ctypes.c_void_p(16), 4, 1000, 1.0,
                                   ctypes.c_void_p(16), None, None) == L.LEAP_ERR_INVALID_ARG
    assert lib.leap_token_logprobs(ctypes.c_void_p(18), 1008, ctypes.c_void_p(16), 4, 1000, 1.0,
                                   ctypes.c_void_p(16), None, None) == L.LEAP_ERR_INVALID_ARG
    lp = L.LossParams(0.2, 0.2, 0.0, 1.0, 0)                  # inv_temp = 0
    assert lib.leap_grpo_loss_fwd(ctypes.byref(lp), ctypes.c_void_p(256), 1024, ctypes.c_void_p(256),
                                  ctypes.c_void_p(256), ctypes.c_void_p(256), ctypes.c_void_p(256), 4, 1024,
                                  ctypes.c_void_p(256), None, None, None, None, ctypes.c_void_p(256), 1 << 20,
                                  None, None) == L.LEAP_ERR_INVALID_ARG
    lp = L.LossParams(0.2, 0.2, 1.0, 1.0, 0)                  # workspace too small
    assert lib.leap_grpo_loss_fwd(ctypes.byref(lp), ctypes.c_void_p(256), 1024, ctypes.c_void_p(256),
                                  ctypes.c_void_p(256), ctypes.c_void_p(256), ctypes.c_void_p(256), 4096, 1024,
                                  ctypes.c_void_p(256), None, None, None, None, ctypes.c_void_p(256), 16,
                                  None, None) == L.LEAP_ERR_INVALID_ARG
    assert lib.leap_grpo_loss_workspace_size(4096, 151936) >= 4096 * 13
    assert lib.leap_selftest_bounded_wait(10, None, None) == L.LEAP_ERR_INVALID_ARG   # limit below 1 us
