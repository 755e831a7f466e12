"""Thin Python binding of libleap (include/leap.h): argument marshalling only.

Every function here has the name of the C entry point it calls, takes torch
CUDA tensors, passes their device pointers and the current CUDA stream, and
raises LeapError on a non-OK status.  All arithmetic runs in libleap's
kernels; there is no fallback: if libleap.so is missing, loading fails.
"""

from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libleap.so")

LEAP_OK = 0
LEAP_ERR_INVALID_ARG = 1
LEAP_ERR_UNSUPPORTED = 2
LEAP_ERR_CUDA = 3
LEAP_ERR_TIMEOUT = 4
LEAP_ERR_BAD_INDEX = 5

LEAP_DEV_BAD_ID = 1
LEAP_DEV_BAD_OUTCOME = 2
LEAP_DEV_BAD_SEGMENT = 4
LEAP_DEV_TIMEOUT = 8

LEAP_CMP_PAPER = 0
LEAP_CMP_LEXI = 1
LEAP_ADVNORM_GRPO_STD = 0
LEAP_ADVNORM_NONE = 1
LEAP_REWARD_RANK = 0
LEAP_REWARD_STATIC = 1
LEAP_AGG_SEQ_MEAN_TOKEN_MEAN = 0
LEAP_AGG_TOKEN_MEAN = 1
LEAP_LOSS_ACCUMULATE = 1
LEAP_LOSS_SINGLE_READ = 2
LEAP_LOSS_INTERLEAVED_ROWS = 4
LEAP_LMHEAD_DHIDDEN = 1
LEAP_LMHEAD_DW = 2
LEAP_PASS_BUCKETS = 10

# Every symbol include/leap.h declares.
EXPORTS = (
    "leap_status_string", "leap_version", "leap_get_device_status",
    "leap_group_rank_advantages", "leap_rollout_token_counts", "leap_scatter_turn_advantages",
    "leap_token_advantages",
    "leap_token_logprobs", "leap_grpo_loss_workspace_size", "leap_grpo_loss_fwd", "leap_grpo_loss_bwd",
    "leap_grpo_loss_fwd_noalloc", "leap_gemm_bf16_nt", "leap_gemm_bf16_tn_f32", "leap_fused_lmhead_workspace_size",
    "leap_fused_lmhead_logprobs", "leap_selftest_bounded_wait",
)
LEAP_NOALLOC_MAX_ROWS = 65536


class LeapError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s returned %s" % (where, status_string(status)))


class RankParams(ctypes.Structure):
    _fields_ = [("num_groups", ctypes.c_int32), ("G", ctypes.c_int32), ("M", ctypes.c_int32),
                ("tau_min", ctypes.c_int32), ("tau_max", ctypes.c_int32), ("gamma", ctypes.c_float),
                ("eps_std", ctypes.c_float), ("cmp", ctypes.c_int32), ("norm", ctypes.c_int32),
                ("std_unbiased", ctypes.c_int32), ("reward", ctypes.c_int32), ("static_c", ctypes.c_float)]


class RankStats(ctypes.Structure):
    _fields_ = [("groups", ctypes.c_int64), ("gated_groups", ctypes.c_int64), ("rollouts", ctypes.c_int64),
                ("nonzero_adv_rollouts", ctypes.c_int64), ("first_turn_passes", ctypes.c_int64),
                ("later_passes", ctypes.c_int64), ("groups_with_recovery", ctypes.c_int64),
                ("failed_first_turn_in_gated", ctypes.c_int64), ("total_turns", ctypes.c_int64),
                ("passes_by_turn", ctypes.c_int64 * 8),
                ("composition", ctypes.c_int64 * (LEAP_PASS_BUCKETS * 3 * 2)),
                ("groups_by_bucket", ctypes.c_int64 * LEAP_PASS_BUCKETS)]


class LossParams(ctypes.Structure):
    _fields_ = [("eps_low", ctypes.c_float), ("eps_high", ctypes.c_float), ("inv_temp", ctypes.c_float),
                ("grad_scale", ctypes.c_float), ("flags", ctypes.c_uint32)]


class LossStats(ctypes.Structure):
    _fields_ = [("loss_sum", ctypes.c_double), ("rho_sum", ctypes.c_double),
                ("live_tokens", ctypes.c_int64), ("clipped_tokens", ctypes.c_int64)]


_lib = None
_P = ctypes.c_void_p
_I32, _I64, _F32, _SZ = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t


def lib() -> ctypes.CDLL:
    """Loads libleap.so (built by paper_2608_01804_gb300.build); fails loudly if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError("libleap.so not found at %s: build it with paper_2608_01804_gb300.build.build()"
                          % LIB_PATH)
    L = ctypes.CDLL(LIB_PATH)
    S = ctypes.c_int  # leap_status_t
    L.leap_status_string.restype = ctypes.c_char_p
    L.leap_status_string.argtypes = [S]
    L.leap_version.restype = _I32
    L.leap_version.argtypes = []
    L.leap_get_device_status.restype = S
    L.leap_get_device_status.argtypes = [ctypes.POINTER(ctypes.c_uint32), _P]
    L.leap_group_rank_advantages.restype = S
    L.leap_group_rank_advantages.argtypes = [ctypes.POINTER(RankParams)] + [_P] * 15
    L.leap_rollout_token_counts.restype = S
    L.leap_rollout_token_counts.argtypes = [_I64, _I32, _I32, _P, _P, _P, _I32, _P, _P, _P, _P]
    L.leap_scatter_turn_advantages.restype = S
    L.leap_scatter_turn_advantages.argtypes = [_I64, _I32, _I32, _P, _P, _P, _I32, _P, _P, _P, _P, _I32,
                                               _P, _P, _P]
    L.leap_token_advantages.restype = S
    L.leap_token_advantages.argtypes = [_I64, _I32, _I32, _P, _P, _P, _I32, _P, _P, _I32, _P, _P, _P, _P, _P]
    L.leap_token_logprobs.restype = S
    L.leap_token_logprobs.argtypes = [_P, _I64, _P, _I64, _I32, _F32, _P, _P, _P]
    L.leap_grpo_loss_workspace_size.restype = _SZ
    L.leap_grpo_loss_workspace_size.argtypes = [_I64, _I32]
    L.leap_grpo_loss_fwd.restype = S
    L.leap_grpo_loss_fwd.argtypes = [ctypes.POINTER(LossParams), _P, _I64, _P, _P, _P, _P, _I64, _I32,
                                     _P, _P, _P, _P, _P, _P, _SZ, _P, _P]
    L.leap_grpo_loss_fwd_noalloc.restype = S
    L.leap_grpo_loss_fwd_noalloc.argtypes = [ctypes.POINTER(LossParams), _P, _I64, _P, _P, _P, _P, _I64, _I32,
                                             _P, _P, _P, _P, _P, _P, _P]
    L.leap_gemm_bf16_nt.restype = S
    L.leap_gemm_bf16_nt.argtypes = [_P, _I64, _P, _I64, _P, _I64, _I32, _I32, _I32, _P]
    L.leap_gemm_bf16_tn_f32.restype = S
    L.leap_gemm_bf16_tn_f32.argtypes = [_P, _I64, _P, _I64, _P, _I64, _I32, _I32, _I32, _I32, _P]
    L.leap_fused_lmhead_workspace_size.restype = _SZ
    L.leap_fused_lmhead_workspace_size.argtypes = [_I64, _I32, _I32, _I32]
    L.leap_fused_lmhead_logprobs.restype = S
    L.leap_fused_lmhead_logprobs.argtypes = [ctypes.POINTER(LossParams), _P, _P, _I64, _I32, _I32, _P, _P, _P, _P,
                                             _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P]
    L.leap_selftest_bounded_wait.restype = S
    L.leap_selftest_bounded_wait.argtypes = [ctypes.c_uint64, _P, _P]
    L.leap_grpo_loss_bwd.restype = S
    L.leap_grpo_loss_bwd.argtypes = [ctypes.POINTER(LossParams), _P, _I64, _P, _P, _P, _P, _P, _I64, _I32,
                                     _P, _P]
    _lib = L
    return L


def status_string(status: int) -> str:
    return lib().leap_status_string(int(status)).decode()


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libleap takes CUDA tensors")
    if not t.is_contiguous():
        raise ValueError("libleap takes contiguous tensors")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(status, where):
    if status != LEAP_OK:
        raise LeapError(status, where)


def _empty(shape, dtype, like):
    return torch.empty(shape, dtype=dtype, device=like.device)


# ---------------------------------------------------------------------------
def leap_get_device_status(stream=None) -> int:
    """Reads and clears the sticky device status bits (synchronises the stream)."""
    v = ctypes.c_uint32(0)
    st = lib().leap_get_device_status(ctypes.byref(v), _stream(stream))
    if st not in (LEAP_OK, LEAP_ERR_BAD_INDEX):
        raise LeapError(st, "leap_get_device_status")
    return int(v.value)


def leap_group_rank_advantages(pass_turn, num_turns, *, G, M, tau_min=0, tau_max=None, gamma=1.0,
                               eps_std=1e-6, norm=LEAP_ADVNORM_GRPO_STD, std_unbiased=True,
                               cmp=LEAP_CMP_PAPER, speedup=None, ntokens=None, gate_in=None, out=None,
                               reward=LEAP_REWARD_RANK, static_c=0.5, stats=None, stream=None):
    """pass_turn, num_turns: int8 [num_groups * G].  Returns a dict of output tensors."""
    n = pass_turn.numel()
    if n % G:
        raise ValueError("pass_turn size is not a multiple of G")
    num_groups = n // G
    if tau_max is None:
        tau_max = G
    if out is None:
        out = dict(gate=_empty(num_groups, torch.uint8, pass_turn), r=_empty(n, torch.uint8, pass_turn),
                   n_worse=_empty(n, torch.int32, pass_turn), n_better=_empty(n, torch.int32, pass_turn),
                   R=_empty(n, torch.float32, pass_turn), A=_empty(n, torch.float32, pass_turn),
                   turn_adv=_empty(n * M, torch.float32, pass_turn), T_eff=_empty(n, torch.uint8, pass_turn))
    p = RankParams(num_groups, G, M, tau_min, tau_max, gamma, eps_std, cmp, norm, 1 if std_unbiased else 0,
                   reward, static_c)
    st = lib().leap_group_rank_advantages(
        ctypes.byref(p), _ptr(pass_turn), _ptr(num_turns), _ptr(speedup), _ptr(ntokens), _ptr(gate_in),
        _ptr(out.get("gate")), _ptr(out.get("r")), _ptr(out.get("n_worse")), _ptr(out.get("n_better")),
        _ptr(out.get("R")), _ptr(out.get("A")), _ptr(out["turn_adv"]), _ptr(out["T_eff"]), _ptr(stats),
        _stream(stream))
    _check(st, "leap_group_rank_advantages")
    return out


def leap_rollout_token_counts(N, seg_offsets, seg_rollout, seg_turn, T_eff, *, M, L=None, totals=None,
                              stream=None):
    """Returns (L int32 [n_rollouts], totals int64 [2])."""
    n = T_eff.numel()
    if L is None:
        L = _empty(n, torch.int32, T_eff)
    if totals is None:
        totals = _empty(2, torch.int64, T_eff)
    st = lib().leap_rollout_token_counts(int(N), n, M, _ptr(seg_offsets), _ptr(seg_rollout), _ptr(seg_turn),
                                         seg_rollout.numel(), _ptr(T_eff), _ptr(L), _ptr(totals),
                                         _stream(stream))
    _check(st, "leap_rollout_token_counts")
    return L, totals


def leap_scatter_turn_advantages(N, seg_offsets, seg_rollout, seg_turn, turn_adv, T_eff, L, totals, *, M,
                                 agg=LEAP_AGG_SEQ_MEAN_TOKEN_MEAN, adv=None, w=None, stream=None):
    """Returns (adv f32 [N], w f32 [N])."""
    if adv is None:
        adv = _empty(int(N), torch.float32, turn_adv)
    if w is None:
        w = _empty(int(N), torch.float32, turn_adv)
    st = lib().leap_scatter_turn_advantages(int(N), T_eff.numel(), M, _ptr(seg_offsets), _ptr(seg_rollout),
                                            _ptr(seg_turn), seg_rollout.numel(), _ptr(turn_adv), _ptr(T_eff),
                                            _ptr(L), _ptr(totals), agg, _ptr(adv), _ptr(w), _stream(stream))
    _check(st, "leap_scatter_turn_advantages")
    return adv, w


def leap_token_advantages(N, seg_offsets, seg_rollout, seg_turn, turn_adv, T_eff, *, M,
                          agg=LEAP_AGG_SEQ_MEAN_TOKEN_MEAN, L=None, totals=None, adv=None, w=None, stream=None):
    """Counts and scatter with the local totals in one call.  Returns (L, totals, adv, w)."""
    n = T_eff.numel()
    L = _empty(n, torch.int32, T_eff) if L is None else L
    totals = _empty(2, torch.int64, T_eff) if totals is None else totals
    adv = _empty(int(N), torch.float32, turn_adv) if adv is None else adv
    w = _empty(int(N), torch.float32, turn_adv) if w is None else w
    st = lib().leap_token_advantages(int(N), n, M, _ptr(seg_offsets), _ptr(seg_rollout), _ptr(seg_turn),
                                     seg_rollout.numel(), _ptr(turn_adv), _ptr(T_eff), agg, _ptr(L), _ptr(totals),
                                     _ptr(adv), _ptr(w), _stream(stream))
    _check(st, "leap_token_advantages")
    return L, totals, adv, w


def _logits_args(logits, V):
    if logits.dtype != torch.bfloat16 or logits.dim() != 2:
        raise ValueError("logits must be a 2-D bf16 tensor")
    if logits.stride(1) != 1:
        raise ValueError("logits rows must be contiguous")
    ld = logits.stride(0)
    if V is None:
        V = logits.shape[1]
    return ctypes.c_void_p(logits.data_ptr()), ld, V


def leap_token_logprobs(logits, ids, *, V=None, inv_temp=1.0, logp=None, lse=None, want_lse=True, stream=None):
    """Returns (logp f32 [N], lse f32 [N] or None)."""
    lp, ld, V = _logits_args(logits, V)
    N = logits.shape[0]
    if logp is None:
        logp = _empty(N, torch.float32, logits)
    if lse is None and want_lse:
        lse = _empty(N, torch.float32, logits)
    st = lib().leap_token_logprobs(lp, ld, _ptr(ids), N, V, inv_temp, _ptr(logp), _ptr(lse), _stream(stream))
    _check(st, "leap_token_logprobs")
    return logp, lse


def leap_grpo_loss_workspace_size(N, V) -> int:
    return int(lib().leap_grpo_loss_workspace_size(int(N), int(V)))


def loss_workspace(N, V, device):
    """A workspace tensor for leap_grpo_loss_fwd (256-byte aligned by the caching allocator)."""
    return torch.empty(max(1, leap_grpo_loss_workspace_size(N, V)), dtype=torch.uint8, device=device)


def leap_grpo_loss_fwd(logits, ids, old_logp, adv, w, *, V=None, eps_low=0.2, eps_high=0.2, inv_temp=1.0,
                       grad_scale=1.0, accumulate=False, loss=None, logp=None, lse=None, ell=None,
                       dlogits=None, want_dlogits=True, want_outputs=True, workspace=None, stats=None,
                       single_read=False, interleaved_rows=False, stream=None):
    """Clipped-surrogate loss (and fused dlogits).  Returns a dict of tensors."""
    lp, ld, V = _logits_args(logits, V)
    N = logits.shape[0]
    if loss is None:
        loss = torch.zeros(1, dtype=torch.float32, device=logits.device)
    if want_outputs:
        logp = _empty(N, torch.float32, logits) if logp is None else logp
        lse = _empty(N, torch.float32, logits) if lse is None else lse
        ell = _empty(N, torch.float32, logits) if ell is None else ell
    if dlogits is None and want_dlogits:
        dlogits = torch.empty_like(logits)
    if workspace is None:
        workspace = loss_workspace(N, V, logits.device)
    flags = ((LEAP_LOSS_ACCUMULATE if accumulate else 0) | (LEAP_LOSS_SINGLE_READ if single_read else 0) |
             (LEAP_LOSS_INTERLEAVED_ROWS if interleaved_rows else 0))
    p = LossParams(eps_low, eps_high, inv_temp, grad_scale, flags)
    st = lib().leap_grpo_loss_fwd(ctypes.byref(p), lp, ld, _ptr(ids), _ptr(old_logp), _ptr(adv), _ptr(w), N, V,
                                  _ptr(loss), _ptr(logp), _ptr(lse), _ptr(ell),
                                  None if dlogits is None else ctypes.c_void_p(dlogits.data_ptr()),
                                  _ptr(workspace), workspace.numel(), _ptr(stats), _stream(stream))
    _check(st, "leap_grpo_loss_fwd")
    return dict(loss=loss, logp=logp, lse=lse, ell=ell, dlogits=dlogits)


def leap_grpo_loss_fwd_noalloc(logits, ids, old_logp, adv, w, *, V=None, eps_low=0.2, eps_high=0.2,
                               inv_temp=1.0, grad_scale=1.0, accumulate=False, loss=None, logp=None, lse=None,
                               ell=None, dlogits=None, want_dlogits=True, want_outputs=True, stats=None,
                               stream=None):
    """leap_grpo_loss_fwd whose scratch is libleap's own device array (no workspace
    argument, N <= LEAP_NOALLOC_MAX_ROWS).  The output tensors are still the caller's."""
    lp, ld, V = _logits_args(logits, V)
    N = logits.shape[0]
    if loss is None:
        loss = torch.zeros(1, dtype=torch.float32, device=logits.device)
    if want_outputs:
        logp = _empty(N, torch.float32, logits) if logp is None else logp
        lse = _empty(N, torch.float32, logits) if lse is None else lse
        ell = _empty(N, torch.float32, logits) if ell is None else ell
    if dlogits is None and want_dlogits:
        dlogits = torch.empty_like(logits)
    p = LossParams(eps_low, eps_high, inv_temp, grad_scale, LEAP_LOSS_ACCUMULATE if accumulate else 0)
    st = lib().leap_grpo_loss_fwd_noalloc(ctypes.byref(p), lp, ld, _ptr(ids), _ptr(old_logp), _ptr(adv), _ptr(w),
                                          N, V, _ptr(loss), _ptr(logp), _ptr(lse), _ptr(ell),
                                          None if dlogits is None else ctypes.c_void_p(dlogits.data_ptr()),
                                          _ptr(stats), _stream(stream))
    _check(st, "leap_grpo_loss_fwd_noalloc")
    return dict(loss=loss, logp=logp, lse=lse, ell=ell, dlogits=dlogits)


def leap_grpo_loss_bwd(logits, ids, old_logp, adv, w, lse, *, V=None, eps_low=0.2, eps_high=0.2, inv_temp=1.0,
                       grad_scale=1.0, dlogits=None, stream=None):
    lp, ld, V = _logits_args(logits, V)
    N = logits.shape[0]
    if dlogits is None:
        dlogits = torch.empty_like(logits)
    p = LossParams(eps_low, eps_high, inv_temp, grad_scale, 0)
    st = lib().leap_grpo_loss_bwd(ctypes.byref(p), lp, ld, _ptr(ids), _ptr(old_logp), _ptr(adv), _ptr(w),
                                  _ptr(lse), N, V, ctypes.c_void_p(dlogits.data_ptr()), _stream(stream))
    _check(st, "leap_grpo_loss_bwd")
    return dlogits


def stats_tensor(device):
    """Device buffer laid out as leap_loss_stats_t (zeroed)."""
    return torch.zeros(ctypes.sizeof(LossStats), dtype=torch.uint8, device=device)


def read_stats(t) -> dict:
    raw = bytes(t.cpu().numpy().tobytes())
    s = LossStats.from_buffer_copy(raw)
    return dict(loss_sum=s.loss_sum, rho_sum=s.rho_sum, live_tokens=s.live_tokens,
                clipped_tokens=s.clipped_tokens)


def _bf16_2d(t, name):
    if t.dtype != torch.bfloat16 or t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("%s must be a 2-D bf16 tensor with contiguous rows" % name)
    return ctypes.c_void_p(t.data_ptr()), t.stride(0)


def leap_gemm_bf16_nt(A, B, out=None, stream=None):
    """out[M x N] = A[M x K] . B[N x K]^T (bf16 in and out, fp32 accumulation on tcgen05)."""
    pa, lda = _bf16_2d(A, "A")
    pb, ldb = _bf16_2d(B, "B")
    M, K = A.shape
    N = B.shape[0]
    if B.shape[1] != K:
        raise ValueError("inner dimensions differ")
    if out is None:   # rows padded to a multiple of 8 elements (16 bytes), returned as an [M x N] view
        out = torch.empty((M, (N + 7) // 8 * 8), dtype=torch.bfloat16, device=A.device)[:, :N]
    pc, ldc = _bf16_2d(out, "out")
    st = lib().leap_gemm_bf16_nt(pa, lda, pb, ldb, pc, ldc, M, N, K, _stream(stream))
    _check(st, "leap_gemm_bf16_nt")
    return out


def leap_gemm_bf16_tn_f32(A, B, out=None, accumulate=False, stream=None):
    """out[M x N] (+)= A[K x M]^T . B[K x N] (bf16 in, fp32 accumulation on tcgen05, fp32 out)."""
    pa, lda = _bf16_2d(A, "A")
    pb, ldb = _bf16_2d(B, "B")
    K, M = A.shape
    N = B.shape[1]
    if B.shape[0] != K:
        raise ValueError("contracted dimensions differ")
    if out is None:   # rows padded to a multiple of 4 elements (16 bytes), returned as an [M x N] view
        out = torch.empty((M, (N + 3) // 4 * 4), dtype=torch.float32, device=A.device)[:, :N]
    if out.dtype != torch.float32 or out.dim() != 2 or out.stride(1) != 1:
        raise ValueError("out must be a 2-D fp32 tensor with contiguous rows")
    st = lib().leap_gemm_bf16_tn_f32(pa, lda, pb, ldb, ctypes.c_void_p(out.data_ptr()), out.stride(0), M, N, K,
                                     1 if accumulate else 0, _stream(stream))
    _check(st, "leap_gemm_bf16_tn_f32")
    return out


def leap_fused_lmhead_workspace_size(N, H, V, with_dhidden=True, with_dW=False) -> int:
    grads = (LEAP_LMHEAD_DHIDDEN if with_dhidden else 0) | (LEAP_LMHEAD_DW if with_dW else 0)
    return int(lib().leap_fused_lmhead_workspace_size(int(N), int(H), int(V), grads))


def leap_fused_lmhead_logprobs(hidden, W, ids, old_logp, adv, w, *, eps_low=0.2, eps_high=0.2, inv_temp=1.0,
                               grad_scale=1.0, accumulate=False, want_dhidden=True, want_dW=False, loss=None,
                               logp=None, lse=None, ell=None, dhidden=None, dW=None, workspace=None, stats=None,
                               stream=None):
    """Clipped-surrogate loss from hidden states and the lm-head weight (logits never stored),
    with the gradients for hidden (bf16) and, if asked, W (fp32; added into `dW` with accumulate)."""
    ph, ldh = _bf16_2d(hidden, "hidden")
    pw, ldw = _bf16_2d(W, "W")
    N, H = hidden.shape
    V = W.shape[0]
    if ldh != H or ldw != H or W.shape[1] != H:
        raise ValueError("hidden and W must be contiguous [N x H] and [V x H]")
    dev = hidden.device
    if loss is None:
        loss = torch.zeros(1, dtype=torch.float32, device=dev)
    logp = _empty(N, torch.float32, hidden) if logp is None else logp
    lse = _empty(N, torch.float32, hidden) if lse is None else lse
    ell = _empty(N, torch.float32, hidden) if ell is None else ell
    if want_dhidden and dhidden is None:
        dhidden = torch.empty_like(hidden)
    if not want_dhidden:
        dhidden = None
    if want_dW and dW is None:
        dW = torch.zeros((V, H), dtype=torch.float32, device=dev)
    if not want_dW:
        dW = None
    if dW is not None and (dW.dtype != torch.float32 or tuple(dW.shape) != (V, H) or not dW.is_contiguous()):
        raise ValueError("dW must be a contiguous fp32 [V x H] tensor")
    if workspace is None:
        workspace = torch.empty(max(1, leap_fused_lmhead_workspace_size(N, H, V, want_dhidden, want_dW)),
                                dtype=torch.uint8, device=dev)
    p = LossParams(eps_low, eps_high, inv_temp, grad_scale, LEAP_LOSS_ACCUMULATE if accumulate else 0)
    st = lib().leap_fused_lmhead_logprobs(ctypes.byref(p), ph, pw, N, H, V, _ptr(ids), _ptr(old_logp), _ptr(adv),
                                          _ptr(w), _ptr(loss), _ptr(logp), _ptr(lse), _ptr(ell),
                                          None if dhidden is None else ctypes.c_void_p(dhidden.data_ptr()),
                                          None if dW is None else ctypes.c_void_p(dW.data_ptr()),
                                          _ptr(workspace), workspace.numel(), _ptr(stats), _stream(stream))
    _check(st, "leap_fused_lmhead_logprobs")
    return dict(loss=loss, logp=logp, lse=lse, ell=ell, dhidden=dhidden, dW=dW)


def rank_stats_tensor(device):
    """Zeroed device buffer laid out as leap_rank_stats_t (the counters accumulate)."""
    return torch.zeros(ctypes.sizeof(RankStats), dtype=torch.uint8, device=device)


def read_rank_stats(t) -> dict:
    """The counters as a dict; 'composition' is nested [bucket][type][sign]."""
    s = RankStats.from_buffer_copy(bytes(t.cpu().numpy().tobytes()))
    arrays = ("passes_by_turn", "composition", "groups_by_bucket")
    d = {k: getattr(s, k) for k, _ in RankStats._fields_ if k not in arrays}
    d["passes_by_turn"] = list(s.passes_by_turn)
    flat = list(s.composition)
    d["composition"] = [[flat[(b * 3 + k) * 2:(b * 3 + k) * 2 + 2] for k in range(3)]
                        for b in range(LEAP_PASS_BUCKETS)]
    d["groups_by_bucket"] = list(s.groups_by_bucket)
    return d


def leap_selftest_bounded_wait(limit_ns, waited=None, stream=None):
    """Runs the bounded-wait self-test kernel (a wait that can never complete,
    given up after limit_ns); `waited` (uint64 device tensor of one element,
    optional) receives the nanoseconds the wait took."""
    st = lib().leap_selftest_bounded_wait(int(limit_ns), _ptr(waited), _stream(stream))
    _check(st, "leap_selftest_bounded_wait")
    return waited
