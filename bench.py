#!/usr/bin/env python
"""Throughput of one LEAP loss hot-path pass (rank advantages -> per-token
advantages -> clipped GRPO surrogate fwd + fused dlogits) on the single-turn
GRPO workload: 16 prompts x G = 8 rollouts x 256 token slots (32,768 rows),
response lengths U{64..256} (the rest is masked padding), vocabulary 151,936,
bf16 logits ~ N(0, 3^2) with 1% of entries raised by 15, synthetic and seeded.

Prints ONE JSON line (rank 0).  `value` counts valid (response) tokens per
second over all ranks.  Usage:
  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl leap|reference]
Under torchrun each rank runs its own batch (weak scaling); the only exchange
is an all-reduce of the two loss normalisers per step.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "rollout tokens/sec through GRPO loss fwd+bwd (V=151936); % of HBM roofline"
UNIT = "tokens/s"
V = 151936
WORKLOAD = ("single-turn GRPO: 16 prompts x G=8 x 256 token slots = 32,768 rows (response lengths U{64..256}, "
            "rest masked padding), V=151936, bf16 logits N(0,3^2) + 1% spikes of +15, old log-probs = current "
            "+ N(0,0.05^2), clip eps 0.2/0.2, seq-mean-token-mean aggregation")

# dram bytes (read + write) of one fused_loss_pipe_kernel launch on this workload: an ncu capture of the
# kernel built from sources with this SHA-256 on a 4,096-row slice, scaled to the full launch by
# algorithmic bytes (traffic grows in proportion to them); null once the sources change.
KNOWN_TRAFFIC = {"src_sha256": "c28bf4a62f446a1c81dffbbdbc115da7babc9b5707ab07b2e0677fd97b0328c9", "bytes_per_launch": 16187086565}
KERNEL_SOURCES = ("paper_2608_01804_gb300/csrc/loss_pipe.cu", "paper_2608_01804_gb300/csrc/leap_common.cuh",
                  "paper_2608_01804_gb300/csrc/loss_math.cuh", "paper_2608_01804_gb300/csrc/row_math.cuh")


def _src_sha():
    h = hashlib.sha256()
    for p in KERNEL_SOURCES:
        h.update(open(os.path.join(ROOT, p), "rb").read())
    return h.hexdigest()


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["leap", "reference"], default="leap")
    ap.add_argument("--e2e-steps", type=int, default=8)
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-rows", action="store_true", help="skip the per-row measurements")
    ap.add_argument("--lmhead-tokens", type=int, default=0,
                    help="run only the fused lm-head (forward + dhidden) on this many tokens, for profiling captures")
    ap.add_argument("--lmhead-dw", action="store_true", help="with --lmhead-tokens: also the weight gradient dW")
    ap.add_argument("--rank-only", action="store_true",
                    help="run only the rank advantages on 65,536 groups x 64 rollouts (M = 3), for profiling captures")
    ap.add_argument("--tokens-only", action="store_true",
                    help="run only the token counts + scatter on the packed multi-turn batch, for profiling captures")
    ap.add_argument("--tokens-layout", choices=["multiturn", "tiny"], default="multiturn",
                    help="with --tokens-only: the packed multi-turn batch or the small padded one")
    ap.add_argument("--logprobs-only", action="store_true",
                    help="run only the log-probs and the forward-only loss on the single-turn batch, for profiling")
    ap.add_argument("--short-rows", action="store_true",
                    help="run only the fused loss fwd + bwd on short vocabularies (1,024-32,768), default and "
                         "single-read kernel")
    ap.add_argument("--short-case", default="",
                    help="with --short-rows: one case VxROWS (e.g. 1024x131072) instead of the sweep")
    ap.add_argument("--multiturn", action="store_true",
                    help="run only the whole pass on the packed multi-turn DCP workload (chunked)")
    ap.add_argument("--lmhead-vocab", type=int, default=0,
                    help="with --lmhead-tokens: a smaller vocabulary, only for small profiling captures")
    ap.add_argument("--prompts", type=int, default=16,
                    help="prompts per rank (16 = the benchmark workload; fewer only for profiling captures)")
    ap.add_argument("--oracle-configs", action="store_true",
                    help="host only: time the oracle on the other workloads (tiny, multi-turn, tournament, "
                         "lm-head), one JSON line each")
    ap.add_argument("--oracle-config-one", default="", help=argparse.SUPPRESS)
    return ap.parse_args()


def _cpu_model():
    """The host CPU's model name (lscpu), for the record beside the oracle's rate."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return None


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def measured_tensor_peak():
    """Sustained dense bf16 TFLOP/s (the lm-head kernels run for tens of ms)."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        return float(json.load(open(p))["bf16_tflops_sustained"])
    return 1700.0


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


class NvmlClockSampler:
    """Samples of this GPU's SM clock, power and clock-event reasons every
    `interval` seconds from a host thread through NVML (libnvidia-ml, read-only
    queries), so that even a timed region of a few tens of milliseconds gets
    several samples.  Raises OSError where NVML cannot be loaded."""

    REASONS = ((0x8, "hw_slowdown"), (0x40, "hw_thermal_slowdown"), (0x20, "sw_thermal_slowdown"),
               (0x4, "sw_power_cap"), (0x80, "hw_power_brake_slowdown"))

    def __init__(self, device, interval=0.005):
        import ctypes
        import threading
        self.ct = ctypes
        self.threading = threading
        self.nvml = ctypes.CDLL("libnvidia-ml.so.1")
        if self.nvml.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        uuid = str(torch.cuda.get_device_properties(device).uuid)
        if not uuid.startswith("GPU-"):
            uuid = "GPU-" + uuid
        self.h = ctypes.c_void_p()
        if self.nvml.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(self.h)) != 0:
            raise OSError("no NVML handle for " + uuid)
        self.reasons_fn = getattr(self.nvml, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(self.nvml, "nvmlDeviceGetCurrentClocksThrottleReasons")
        self.interval = interval
        self.samples = []
        self.stop_evt = threading.Event()
        self.thread = None
        self.max_mhz = self._uint(self.nvml.nvmlDeviceGetMaxClockInfo, 1)

    def _uint(self, fn, *args):
        v = self.ct.c_uint(0)
        return v.value if fn(self.h, *args, self.ct.byref(v)) == 0 else None

    def _sample(self):
        sm = self._uint(self.nvml.nvmlDeviceGetClockInfo, 1)
        mw = self._uint(self.nvml.nvmlDeviceGetPowerUsage)
        r = self.ct.c_ulonglong(0)
        reasons = r.value if self.reasons_fn(self.h, self.ct.byref(r)) == 0 else 0
        if sm is not None:
            self.samples.append((sm, mw, reasons))

    def _run(self):
        while not self.stop_evt.is_set():
            self._sample()
            self.stop_evt.wait(self.interval)

    def start(self):
        self.samples = []
        self.stop_evt.clear()
        self.thread = self.threading.Thread(target=self._run, daemon=True)
        self.thread.start()

    def stop(self):
        self.stop_evt.set()
        self.thread.join()
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": ["no samples"], "source": "nvml"}
        reasons = sorted({nm for _, _, bits in self.samples for b, nm in self.REASONS if bits & b})
        power = [mw / 1000.0 for _, mw, _ in self.samples if mw is not None]
        return {"sm_mhz": statistics.median(sm for sm, _, _ in self.samples), "sm_max_mhz": self.max_mhz,
                "samples": len(self.samples), "power_w_max": max(power) if power else None, "reasons": reasons,
                "source": "nvml, %g ms interval" % (1000 * self.interval)}


def clock_sampler(device):
    """NVML sampling where the library loads, else nvidia-smi."""
    try:
        return NvmlClockSampler(device)
    except (OSError, AttributeError):
        return ClockSampler(device)


class ClockSampler:
    """nvidia-smi samples of this GPU's clocks and throttle reasons every 200 ms."""

    FIELDS = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        try:
            self.uuid = str(torch.cuda.get_device_properties(device).uuid)
        except Exception:
            self.uuid = None
        self.proc = None

    def start(self):
        self.out = tempfile.NamedTemporaryFile(mode="w+", suffix=".csv", delete=False)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait()
        self.out.flush()
        self.out.seek(0)
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.out.read().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            if self.uuid and self.uuid not in f[0] and f[0] not in self.uuid:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
                power.append(float(f[3]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        os.unlink(self.out.name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "samples": len(sm),
                "power_w_max": max(power), "reasons": sorted(reasons)}


def torch_logp(logits, ids, chunk=2048):
    """Current-policy log-probs with torch's fp32 log_softmax: input generation of
    the old log-probs only (outside every timed region)."""
    out = torch.empty(logits.shape[0], dtype=torch.float32, device=logits.device)
    for a in range(0, logits.shape[0], chunk):
        b = min(logits.shape[0], a + chunk)
        out[a:b] = torch.log_softmax(logits[a:b].float(), dim=1).gather(1, ids[a:b].long().view(-1, 1)).view(-1)
    return out


def make_inputs(rank, device, prompts=16):
    from paper_2608_01804_gb300 import synth
    batch = synth.single_turn_batch(seed=1 + 1000 * rank, num_prompts=prompts)
    N = batch.N
    logits = synth.logits(N, V, 3.0, 200 + rank, device, spike_frac=0.01)
    ids = synth.token_ids(N, V, 201 + rank, device)
    old = torch_logp(logits, ids) + synth.normal(N, 0.05, 202 + rank, device)
    return batch, logits, ids, old


def valid_tokens(batch):
    return int(sum(int(batch.seg_offsets[s + 1] - batch.seg_offsets[s])
                   for s in range(len(batch.seg_rollout)) if batch.seg_turn[s] >= 0))


def cpu_oracle_rate(batch, logits, ids, old, seconds, block=32):
    """The oracle as it stands on a bounded sample of the same workload: the
    rank/token steps on the whole batch, then the loss fwd + dlogits over rows
    in order until `seconds` of CPU time; returns (valid tokens/s, rows, valid)."""
    from oracle import leap_oracle as O
    G, M = batch.G, batch.M
    t_total = 0.0
    t0 = time.perf_counter()
    orc = O.rank_advantages(batch.pass_turn.reshape(-1, G), batch.num_turns.reshape(-1, G), M, 0, G, 1.0)
    ta, te = orc["turn_adv"].reshape(-1), orc["T_eff"].reshape(-1)
    Lc, nv, rv = O.rollout_token_counts(batch.seg_offsets, batch.seg_rollout, batch.seg_turn, te)
    adv, w = O.token_advantages(batch.N, batch.seg_offsets, batch.seg_rollout, batch.seg_turn, ta, te, M, 0, Lc, nv, rv)
    t_total += time.perf_counter() - t0
    rows = valid = 0
    ids_h = ids.cpu().numpy().astype(np.int64)
    old_h = old.cpu().numpy().astype(np.float64)
    while t_total < seconds and rows < batch.N:
        a, b = rows, min(batch.N, rows + block)
        bits = logits[a:b].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        z = O.bf16_bits_to_f64(bits)
        t0 = time.perf_counter()
        O.grpo_loss_rows(z, ids_h[a:b], old_h[a:b], adv[a:b], w[a:b])
        t_total += time.perf_counter() - t0
        valid += int(np.count_nonzero(w[a:b]))
        rows = b
    return valid / t_total, rows, valid, t_total


# ---- the oracle on every host core (a process pool started with spawn) ----
_SHM = {}


def _pool_init(shm_name, shape):
    """Worker start-up: one thread per worker, attach the shared logits bits."""
    from multiprocessing import shared_memory
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[k] = "1"
    shm = shared_memory.SharedMemory(name=shm_name)
    _SHM["shm"] = shm
    _SHM["bits"] = np.ndarray(shape, dtype=np.uint16, buffer=shm.buf)


def _pool_rows(task):
    """The oracle's loss forward and dlogits on rows [a, b) (weights w != 0 only are read)."""
    from oracle import leap_oracle as O
    a, b, ids, old, adv, w = task
    live = np.nonzero(w)[0]
    if len(live) == 0:
        return 0
    z = O.bf16_bits_to_f64(_SHM["bits"][a:b][live])
    O.grpo_loss_rows(z, ids[live], old[live], adv[live], w[live])
    return len(live)


def cpu_oracle_rate_all_cores(batch, logits, ids, old, block=32):
    """The oracle (as it stands) over the WHOLE batch on every host core: the
    rank/token steps once, then the loss forward + dlogits of every row in
    blocks of `block` rows, spread over os.cpu_count() spawned workers that
    read the bf16 logits from host shared memory.  Returns (valid tokens/s,
    workers, valid tokens, seconds)."""
    import multiprocessing as mp
    from multiprocessing import shared_memory
    from oracle import leap_oracle as O
    G, M = batch.G, batch.M
    N, Vr = logits.shape
    workers = os.cpu_count() or 1
    shm = shared_memory.SharedMemory(create=True, size=N * Vr * 2)
    try:
        bits = np.ndarray((N, Vr), dtype=np.uint16, buffer=shm.buf)
        for a0 in range(0, N, 4096):
            b0 = min(N, a0 + 4096)
            bits[a0:b0] = logits[a0:b0].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        ids_h = ids.cpu().numpy().astype(np.int64)
        old_h = old.cpu().numpy().astype(np.float64)
        ctx = mp.get_context("spawn")
        with ctx.Pool(workers, initializer=_pool_init, initargs=(shm.name, (N, Vr))) as pool:
            pool.map(_pool_rows, [(0, 0, ids_h[:0], old_h[:0], old_h[:0], old_h[:0])] * workers)   # start-up
            t0 = time.perf_counter()
            orc = O.rank_advantages(batch.pass_turn.reshape(-1, G), batch.num_turns.reshape(-1, G), M, 0, G, 1.0)
            ta, te = orc["turn_adv"].reshape(-1), orc["T_eff"].reshape(-1)
            Lc, nv, rv = O.rollout_token_counts(batch.seg_offsets, batch.seg_rollout, batch.seg_turn, te)
            adv, w = O.token_advantages(batch.N, batch.seg_offsets, batch.seg_rollout, batch.seg_turn, ta, te, M, 0,
                                        Lc, nv, rv)
            tasks = [(a, min(N, a + block), ids_h[a:a + block], old_h[a:a + block], adv[a:a + block], w[a:a + block])
                     for a in range(0, N, block)]
            valid = sum(pool.imap_unordered(_pool_rows, tasks, chunksize=1))
            secs = time.perf_counter() - t0
        return valid / secs, workers, valid, secs
    finally:
        shm.close()
        shm.unlink()


def workload_config(prompts, rows, valid, world):
    """The `config` object of both arms' JSON lines."""
    return {"workload": WORKLOAD if prompts == 16 else "%d-prompt slice of: %s" % (prompts, WORKLOAD),
            "rows_per_step_per_gpu": rows, "valid_tokens_per_step_per_gpu": valid,
            "vocab": V, "logits_dtype": "bf16", "l2": "inputs larger than L2 (9.96 GB of logits "
            "read and 9.96 GB of dlogits written per step)", "parallelism": "dp%d" % world}


def _oracle_one(name, seconds):
    """The oracle as it stands on one workload, in this process (its BLAS
    threads as the environment set them); returns the JSON-ready record."""
    from oracle import leap_oracle as O
    from paper_2608_01804_gb300 import synth
    t_begin = time.perf_counter()

    def rank_tokens(batch):
        G, M = batch.G, batch.M
        gate = batch.gate_in
        orc = O.rank_advantages(batch.pass_turn.reshape(-1, G), batch.num_turns.reshape(-1, G), M, 0, G, 0.9,
                                gate_in=gate)
        ta, te = orc["turn_adv"].reshape(-1), orc["T_eff"].reshape(-1)
        Lc, nv, rv = O.rollout_token_counts(batch.seg_offsets, batch.seg_rollout, batch.seg_turn, te)
        return O.token_advantages(batch.N, batch.seg_offsets, batch.seg_rollout, batch.seg_turn, ta, te, M, 0,
                                  Lc, nv, rv)

    def loss_rows(z_bits, ids, old, adv, w):
        live = np.nonzero(w)[0]
        z = O.bf16_bits_to_f64(z_bits[live])
        O.grpo_loss_rows(z, ids[live], old[live], adv[live], w[live])
        return len(live)

    if name == "tiny":          # 16,384 rows at V = 1,024, timed whole
        batch = synth.tiny_batch()
        Vt = 1024
        z = synth.logits(batch.N, Vt, 2.0, 300, "cpu")
        ids = synth.token_ids(batch.N, Vt, 301, "cpu")
        old = (torch_logp(z, ids) + synth.normal(batch.N, 0.05, 302, "cpu")).numpy().astype(np.float64)
        bits = z.view(torch.int16).numpy().view(np.uint16)
        t0 = time.perf_counter()
        adv, w = rank_tokens(batch)
        valid = loss_rows(bits, ids.numpy().astype(np.int64), old, adv, w)
        dt = time.perf_counter() - t0
        return {"config": "tiny: 4 prompts x G=8 x 2 turns x 256 = 16,384 rows, V=1024", "value": valid / dt,
                "unit": "valid tokens/s", "sample": "the whole step (%d valid tokens), %.1f s" % (valid, dt)}
    if name == "multiturn":     # rank/token steps on the whole stream, the loss on a sample of its live rows
        batch = synth.multiturn_dcp_batch()
        src = 256                                   # logits rows drawn once, reused for every row
        z = synth.logits(src, V, 3.0, 310, "cpu", spike_frac=0.01)
        ids_src = synth.token_ids(src, V, 311, "cpu")
        old_src = (torch_logp(z, ids_src) + synth.normal(src, 0.05, 312, "cpu")).numpy().astype(np.float64)
        bits = z.view(torch.int16).numpy().view(np.uint16)
        ids_src = ids_src.numpy().astype(np.int64)
        t0 = time.perf_counter()
        adv, w = rank_tokens(batch)
        t_rt = time.perf_counter() - t0
        live = np.nonzero(w)[0]
        done, t_loss = 0, 0.0
        while t_loss < seconds and done < len(live):
            rows = live[done:done + 32]
            k = rows % src
            t1 = time.perf_counter()
            O.grpo_loss_rows(O.bf16_bits_to_f64(bits[k]), ids_src[k], old_src[k], adv[rows], w[rows])
            t_loss += time.perf_counter() - t1
            done += len(rows)
        est = t_rt + t_loss / done * len(live)
        return {"config": "multi-turn DCP: 32 prompts x G=16, M=3, %d rows (%d valid), V=151936" % (batch.N, len(live)),
                "value": len(live) / est, "unit": "valid tokens/s",
                "sample": "rank/token oracle on the whole stream (%.1f s) + loss fwd and dlogits of the first %d "
                          "valid rows (%.1f s), scaled to all %d" % (t_rt, done, t_loss, len(live))}
    if name == "tournament":    # 65,536 groups x 64, M = 3: groups in order until the time is up
        pt, nt, _, _ = synth.tournament_outcomes()
        G, M = 64, 3
        pt, nt = pt.reshape(-1, G), nt.reshape(-1, G)
        done, dt, step = 0, 0.0, 1024
        while dt < seconds and done < pt.shape[0]:
            t1 = time.perf_counter()
            O.rank_advantages(pt[done:done + step], nt[done:done + step], M, 50, 56, 0.9)
            dt += time.perf_counter() - t1
            done += min(step, pt.shape[0] - done)
        return {"config": "tournament: 65,536 groups x G=64, M=3", "value": done * G / dt, "unit": "rollouts/s",
                "sample": "%d groups in blocks of %d, %.1f s" % (done, step, dt)}
    if name == "lmhead":        # 64 tokens of hidden W^T, loss and dhidden, fp64
        H, T = 5120, 64
        rng = np.random.default_rng(320)
        hidden = rng.standard_normal((T, H))
        Wm = rng.standard_normal((V, H)) * 0.02
        ids = rng.integers(0, V, T)
        old = np.full(T, -12.0)
        adv = rng.standard_normal(T)
        w = np.full(T, 1.0 / T)
        t0 = time.perf_counter()
        O.lmhead_loss_rows(hidden, Wm, ids, old, adv, w, want_dhidden=True)
        dt = time.perf_counter() - t0
        return {"config": "fused lm-head: hidden [65,536 x 5120] x W [151,936 x 5120]", "value": T / dt,
                "unit": "tokens/s (forward + dhidden)",
                "sample": "%d tokens (logits, loss, dlogits, dhidden in fp64), %.1f s; the whole 65,536 would take "
                          "%.0f s" % (T, dt, dt * 65536 / T)}
    raise ValueError(name)


def oracle_configs(args):
    """The oracle, as it stands, on the other workloads: each measurement in a
    fresh process, with one BLAS thread and (the lm-head's matrix products)
    with every core; one JSON line per measurement."""
    cores = os.cpu_count() or 1
    runs = [("tiny", 1), ("multiturn", 1), ("tournament", 1), ("lmhead", 1), ("lmhead", cores)]
    for name, threads in runs:
        env = dict(os.environ)
        for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
            env[k] = str(threads)
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-config-one", name,
                            "--cpu-seconds", str(args.cpu_seconds)], env=env, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("oracle timing %s failed:\n%s" % (name, r.stderr[-2000:]))
        rec = json.loads(r.stdout.strip().splitlines()[-1])
        rec.update({"kind": "oracle", "cores": threads, "cpu_model": _cpu_model()})
        print(json.dumps(rec), flush=True)


def reference_arm(args):
    """The oracle (fp64 CPU) as the reference implementation, timed per step on
    a bounded sample of the same workload; rank 0 only."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from oracle import leap_oracle as O
    from paper_2608_01804_gb300 import synth
    batch = synth.single_turn_batch(seed=1)
    G, M = batch.G, batch.M
    sample = 48                                   # rows of the loss per step
    z_bits = synth.logits(sample * 4, V, 3.0, 200, "cpu", spike_frac=0.01)
    ids = synth.token_ids(sample * 4, V, 201, "cpu")
    old = torch_logp(z_bits, ids) + synth.normal(sample * 4, 0.05, 202, "cpu")
    z = O.bf16_bits_to_f64(z_bits.view(torch.int16).numpy().view(np.uint16))
    ids_h, old_h = ids.numpy().astype(np.int64), old.numpy().astype(np.float64)

    def one_step(k):
        orc = O.rank_advantages(batch.pass_turn.reshape(-1, G), batch.num_turns.reshape(-1, G), M, 0, G, 1.0)
        ta, te = orc["turn_adv"].reshape(-1), orc["T_eff"].reshape(-1)
        Lc, nv, rv = O.rollout_token_counts(batch.seg_offsets, batch.seg_rollout, batch.seg_turn, te)
        adv, w = O.token_advantages(batch.N, batch.seg_offsets, batch.seg_rollout, batch.seg_turn, ta, te, M, 0,
                                    Lc, nv, rv)
        a = (k % 4) * sample
        live = np.nonzero(w)[0][a:a + sample]
        O.grpo_loss_rows(z[a:a + sample], ids_h[a:a + sample], old_h[a:a + sample], adv[live], w[live])
        return len(live)

    for k in range(args.warmup):
        one_step(k)
    t0 = time.perf_counter()
    toks = sum(one_step(k) for k in range(args.steps))
    dt = time.perf_counter() - t0
    value = toks / dt
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": workload_config(16, batch.N, valid_tokens(batch), args.gpus),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": "per step: rank/token oracle on the whole batch + loss fwd and dlogits on "
                                       "%d valid rows" % sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# Rows per host-to-device chunk of the end-to-end leg (1.24 GB of logits at V = 151,936).
E2E_CHUNK_ROWS = 4096

# GPU cycles (~100 us) the stream spins before a short row's start event, so
# that the row's launches are all queued by the time the device reaches them.
LEAD_CYCLES = 200000


def _timed_launches(fn, reps, stream, flush=None, lead_cycles=0):
    """Average device time of fn() over `reps` launches, each timed with CUDA
    events on the launching stream; `flush` (untimed) runs before each.  With
    lead_cycles the stream first spins that many GPU cycles (untimed), so every
    launch of fn() is queued before the start event is reached and the time is
    the device's, not the host's launch latency."""
    total = 0.0
    for _ in range(reps):
        if flush is not None:
            flush()
        if lead_cycles:
            torch.cuda._sleep(lead_cycles)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        b.synchronize()
        total += a.elapsed_time(b)
    return total / reps


MT_CHUNK = 65536   # rows per logits chunk of the multi-turn stream


def multiturn_step(device, peak, steps=3, warmup=1):
    """The whole pass on the packed multi-turn DCP workload (32 prompts x G = 16,
    up to 3 turns, prompts and feedback masked, ~1.49 M rows, V = 151,936)
    through GrpoStep.run_chunked: rank -> counts -> scatter over the whole
    stream, then the fused loss over 65,536-row chunks with loss accumulation.
    The stream's 452 GB of logits exceed HBM, so one 65,536-row chunk of logits
    (19.9 GB, N(0, 3^2) + 1% spikes) is drawn once and stands in for every chunk
    (the ids, old log-probs, advantages and weights are the true per-row ones);
    dlogits go to one chunk buffer likewise.  Each chunk is larger than L2."""
    from paper_2608_01804_gb300 import synth
    from paper_2608_01804_gb300.step import GrpoStep
    b = synth.multiturn_dcp_batch()
    N = b.N
    zbuf = synth.logits(MT_CHUNK, V, 3.0, 300, device, spike_frac=0.01)
    dlbuf = torch.empty_like(zbuf)
    ids = synth.token_ids(N, V, 301, device)
    old = torch.empty(N, dtype=torch.float32, device=device)
    for a in range(0, N, MT_CHUNK):   # current-policy log-probs of each chunk's rows (input generation)
        n = min(MT_CHUNK, N - a)
        old[a:a + n] = torch_logp(zbuf[:n], ids[a:a + n])
    old += synth.normal(N, 0.05, 302, device)
    step = GrpoStep(b, V, device, gamma=0.9, tau=(8, 15), use_gate_in=False, chunk_rows=MT_CHUNK)
    chunks = [(a, zbuf[:min(MT_CHUNK, N - a)], dlbuf[:min(MT_CHUNK, N - a)]) for a in range(0, N, MT_CHUNK)]
    for _ in range(max(1, warmup)):
        step.run_chunked(chunks, ids, old)
    torch.cuda.synchronize()
    live = int((step.w != 0).sum().item())
    tok_launches = step.token_launches()
    stream = torch.cuda.current_stream()
    a_ev, b_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a_ev.record(stream)
    for _ in range(steps):
        step.run_chunked(chunks, ids, old)
    b_ev.record(stream)
    b_ev.synchronize()
    ms = a_ev.elapsed_time(b_ev) / steps
    alg = live * 4 * V + (N - live) * 2 * V + 16 * N
    gbs = alg / (ms / 1e3) / 1e9
    out = {"ms_per_step": ms, "rows": N, "valid_tokens": live, "chunks": len(chunks), "algorithmic_bytes": alg,
           "achieved_gbs": gbs, "frac": gbs / peak, "throughput": live / (ms / 1e3), "unit": "valid tokens/s",
           "launches_per_step": 1 + tok_launches + 3 * len(chunks),
           "note": "whole step (rank, counts, scatter, fused loss + reductions per chunk); one 65,536-row "
                   "logits chunk reused for every chunk"}
    del zbuf, dlbuf, step
    torch.cuda.synchronize()
    return out


def measure_rows(device, logits, ids, old, step, peak, reps=5):
    """Each remaining row of the hot path on its own workload, against the HBM
    roofline: rank advantages on 65,536 groups x 64 rollouts (M = 3), token
    counts + scatter on the packed multi-turn batch, log-probs and the split
    forward / backward on the single-turn batch."""
    from paper_2608_01804_gb300 import leap as L
    from paper_2608_01804_gb300 import synth
    stream = torch.cuda.current_stream()
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=device)   # > L2: evicts between launches
    flush = lambda: flush_buf.fill_(1)
    rows = {}

    def entry(bytes_, ms, unit_count, unit):
        gbs = bytes_ / (ms / 1e3) / 1e9
        return {"ms": ms, "algorithmic_bytes": bytes_, "achieved_gbs": gbs, "frac": gbs / peak,
                "throughput": unit_count / (ms / 1e3), "unit": unit}

    # a1-a3: rank advantages, tournament stress workload.
    pt, nt, _, _ = synth.tournament_outcomes()
    G, M = 64, 3
    n = pt.size
    pt_d = torch.as_tensor(pt).to(device)
    nt_d = torch.as_tensor(nt).to(device)
    out = L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=50, tau_max=56, gamma=0.9)
    fn = lambda: L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=50, tau_max=56, gamma=0.9, out=out)
    fn()
    ms = _timed_launches(fn, reps * 4, stream, flush, lead_cycles=LEAD_CYCLES)
    rank_bytes = n * (2 + 1 + 4 + 4 + 4 + 4 + 4 * M + 1) + n // G
    rows["rank_advantages_65536x64"] = entry(rank_bytes, ms, n, "rollouts/s")
    # The extension modes on the same workload: tie-broken tournament (reads
    # speedup and tokens too), training counters, static-scalar reward.
    _, _, sp, tk = synth.tournament_outcomes()
    sp_d = torch.as_tensor(sp).to(device)
    tk_d = torch.as_tensor(tk).to(device)
    stats = L.rank_stats_tensor(device)
    variants = {
        "rank_advantages_lexi_65536x64": (dict(cmp=L.LEAP_CMP_LEXI, speedup=sp_d, ntokens=tk_d), 8 * n),
        "rank_advantages_with_counters_65536x64": (dict(stats=stats), 0),
        "rank_advantages_static_reward_65536x64": (dict(reward=L.LEAP_REWARD_STATIC, static_c=0.5), 0),
    }
    for name, (kw, extra) in variants.items():
        fv = lambda kw=kw: L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=50, tau_max=56, gamma=0.9,
                                                        out=out, **kw)
        fv()
        ms = _timed_launches(fv, reps * 4, stream, flush, lead_cycles=LEAD_CYCLES)
        rows[name] = entry(rank_bytes + extra, ms, n, "rollouts/s")
    del pt_d, nt_d, out, sp_d, tk_d, stats

    # a4: per-rollout counts + per-token scatter, packed multi-turn batch.
    b = synth.multiturn_dcp_batch()
    pt_d = torch.as_tensor(b.pass_turn).to(device)
    nt_d = torch.as_tensor(b.num_turns).to(device)
    rk = L.leap_group_rank_advantages(pt_d, nt_d, G=b.G, M=b.M, tau_min=8, tau_max=15, gamma=0.9)
    so = torch.as_tensor(b.seg_offsets).to(device)
    sr = torch.as_tensor(b.seg_rollout).to(device)
    st_ = torch.as_tensor(b.seg_turn).to(device)
    Lc, tot = L.leap_rollout_token_counts(b.N, so, sr, st_, rk["T_eff"], M=b.M)
    adv, w = L.leap_scatter_turn_advantages(b.N, so, sr, st_, rk["turn_adv"], rk["T_eff"], Lc, tot, M=b.M)

    def tok():
        L.leap_rollout_token_counts(b.N, so, sr, st_, rk["T_eff"], M=b.M, L=Lc, totals=tot)
        L.leap_scatter_turn_advantages(b.N, so, sr, st_, rk["turn_adv"], rk["T_eff"], Lc, tot, M=b.M, adv=adv, w=w)
    ms = _timed_launches(tok, reps * 4, stream, flush, lead_cycles=LEAD_CYCLES)
    rows["token_counts_scatter_multiturn_%d_tokens" % b.N] = entry(8 * b.N, ms, b.N, "tokens/s")
    fused = lambda: L.leap_token_advantages(b.N, so, sr, st_, rk["turn_adv"], rk["T_eff"], M=b.M, L=Lc, totals=tot,
                                            adv=adv, w=w)
    ms = _timed_launches(fused, reps * 4, stream, flush, lead_cycles=LEAD_CYCLES)
    rows["token_advantages_one_launch_multiturn_%d_tokens" % b.N] = entry(8 * b.N, ms, b.N, "tokens/s")
    # The same two ways on the small workload's padded layout (16,384 tokens).
    tbk = synth.tiny_batch()
    t_so, t_sr, t_st = (torch.as_tensor(x).to(device) for x in (tbk.seg_offsets, tbk.seg_rollout, tbk.seg_turn))
    t_rk = L.leap_group_rank_advantages(torch.as_tensor(tbk.pass_turn).to(device),
                                        torch.as_tensor(tbk.num_turns).to(device), G=tbk.G, M=tbk.M, gamma=0.9)
    t_L, t_tot, t_adv, t_w = L.leap_token_advantages(tbk.N, t_so, t_sr, t_st, t_rk["turn_adv"], t_rk["T_eff"], M=tbk.M)

    def t_two():
        L.leap_rollout_token_counts(tbk.N, t_so, t_sr, t_st, t_rk["T_eff"], M=tbk.M, L=t_L, totals=t_tot)
        L.leap_scatter_turn_advantages(tbk.N, t_so, t_sr, t_st, t_rk["turn_adv"], t_rk["T_eff"], t_L, t_tot,
                                       M=tbk.M, adv=t_adv, w=t_w)
    t_one = lambda: L.leap_token_advantages(tbk.N, t_so, t_sr, t_st, t_rk["turn_adv"], t_rk["T_eff"], M=tbk.M,
                                            L=t_L, totals=t_tot, adv=t_adv, w=t_w)
    ms = _timed_launches(t_two, reps * 4, stream, flush, lead_cycles=LEAD_CYCLES)
    rows["token_counts_scatter_tiny_%d_tokens" % tbk.N] = entry(8 * tbk.N, ms, tbk.N, "tokens/s")
    ms = _timed_launches(t_one, reps * 4, stream, flush, lead_cycles=LEAD_CYCLES)
    rows["token_advantages_one_launch_tiny_%d_tokens" % tbk.N] = entry(8 * tbk.N, ms, tbk.N, "tokens/s")
    del adv, w

    # The whole pass on the multi-turn DCP workload (a1-a7 over the chunked stream).
    rows["multiturn_dcp_step_%d_rows_V151936" % b.N] = multiturn_step(device, peak)

    # a5: log-probs (2V bytes per row), and the split forward / backward (a6, a7).
    N = logits.shape[0]
    logp = torch.empty(N, dtype=torch.float32, device=device)
    lse = torch.empty(N, dtype=torch.float32, device=device)
    fn = lambda: L.leap_token_logprobs(logits, ids, V=V, logp=logp, lse=lse)
    fn()
    ms = _timed_launches(fn, reps, stream)
    rows["token_logprobs_32768xV"] = entry(2 * V * N + 12 * N, ms, N, "tokens/s")
    live = int((step.w != 0).sum().item())
    ws = L.loss_workspace(N, V, device)
    fwd = lambda: L.leap_grpo_loss_fwd(logits, ids, old, step.adv, step.w, V=V, loss=step.loss, lse=lse,
                                       want_dlogits=False, want_outputs=False, workspace=ws)
    fwd()
    ms_f = _timed_launches(fwd, reps, stream)
    rows["loss_fwd_only_32768xV"] = entry(2 * V * live + 16 * N, ms_f, live, "valid tokens/s")
    dl = torch.empty_like(logits)
    bwd = lambda: L.leap_grpo_loss_bwd(logits, ids, old, step.adv, step.w, lse, V=V, dlogits=dl)
    bwd()
    ms_b = _timed_launches(bwd, reps, stream)
    rows["loss_bwd_split_32768xV"] = entry(4 * V * live + 2 * V * (N - live) + 20 * N, ms_b, live, "valid tokens/s")
    split = entry(6 * V * live + 2 * V * (N - live) + 36 * N, ms_f + ms_b, live, "valid tokens/s")
    split["frac_vs_fused_4V_bytes"] = (4 * V * live + 2 * V * (N - live) + 16 * N) / ((ms_f + ms_b) / 1e3) / 1e9 / peak
    rows["split_fwd_then_bwd_32768xV"] = split
    del dl, ws
    torch.cuda.synchronize()

    # The whole pass (a1-a7) on the small workload (4 prompts x 8 x 2 turns x
    # 256 = 16,384 rows, V = 1,024; 32 MB of logits, resident in L2), where the
    # host's launches cost more than the kernels: 100 back-to-back steps
    # launched kernel by kernel, then as replays of one CUDA graph.
    from paper_2608_01804_gb300.step import GrpoStep
    tb = synth.tiny_batch()
    Vt = 1024
    zt = synth.logits(tb.N, Vt, 2.0, 700, device)
    it = synth.token_ids(tb.N, Vt, 701, device)
    ot = torch_logp(zt, it) + synth.normal(tb.N, 0.05, 702, device)
    st_t = GrpoStep(tb, Vt, device, gamma=0.9, tau=(0, tb.G))
    dl_t = torch.empty_like(zt)
    graph = st_t.capture(zt, it, ot, dl_t)

    def back_to_back(fn, k=100):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record(stream)
        for _ in range(k):
            fn()
        b.record(stream)
        b.synchronize()
        return a.elapsed_time(b) / k

    eager_ms = back_to_back(lambda: st_t.run(zt, it, ot, dl_t))
    graph_ms = back_to_back(graph.replay)
    nv_t = int((st_t.w != 0).sum().item())   # weighted tokens: DCP-pruned turns in the layout count none
    rows["step_tiny_16384xV1024_eager_vs_graph"] = {
        "eager_ms": eager_ms, "graph_ms": graph_ms, "launches_per_step": st_t.launches_per_run(),
        "eager_valid_tokens_per_s": nv_t / (eager_ms / 1e3), "graph_valid_tokens_per_s": nv_t / (graph_ms / 1e3),
        "note": "100 back-to-back steps, host launch cost included, logits resident in L2"}
    del graph, st_t, zt, dl_t
    torch.cuda.synchronize()

    # a8: fused lm-head (tcgen05), 65,536 tokens x H = 5,120 x V = 151,936.
    lb = synth.lmhead_batch()
    N8, H = lb.N, 5120
    hidden = synth.normal((N8, H), 1.0, 500, device, dtype=torch.bfloat16)
    W = synth.normal((V, H), 0.02, 501, device, dtype=torch.bfloat16)
    ids8 = synth.token_ids(N8, V, 502, device)
    old8 = torch.empty(N8, dtype=torch.float32, device=device)
    for a0 in range(0, N8, 4096):     # current-policy log-probs (torch), input generation only
        zc = (hidden[a0:a0 + 4096] @ W.T).float()
        old8[a0:a0 + 4096] = torch.log_softmax(zc, 1).gather(1, ids8[a0:a0 + 4096].long().view(-1, 1)).view(-1)
        del zc
    old8 += synth.normal(N8, 0.05, 503, device)
    st8 = GrpoStep(lb, V, device, gamma=1.0, tau=(0, lb.G), use_gate_in=False)
    st8.advantages()
    ws8 = torch.empty(L.leap_fused_lmhead_workspace_size(N8, H, V, True, True), dtype=torch.uint8, device=device)
    dh = torch.empty_like(hidden)
    dW = torch.empty((V, H), dtype=torch.float32, device=device)
    fwd8 = lambda: L.leap_fused_lmhead_logprobs(hidden, W, ids8, old8, st8.adv, st8.w, want_dhidden=False,
                                                workspace=ws8)
    full8 = lambda: L.leap_fused_lmhead_logprobs(hidden, W, ids8, old8, st8.adv, st8.w, dhidden=dh, workspace=ws8)
    fwd8()
    full8()
    tpeak = measured_tensor_peak()
    ms = _timed_launches(fwd8, 3, stream)
    fl = 2.0 * N8 * V * H
    rows["fused_lmhead_fwd_65536x5120xV"] = {"ms": ms, "algorithmic_flops": fl, "achieved_tflops": fl / ms / 1e9,
                                            "frac": fl / ms / 1e9 / tpeak, "throughput": N8 / (ms / 1e3),
                                            "unit": "tokens/s", "bound": "tensor"}
    ms = _timed_launches(full8, 3, stream)
    fl = 6.0 * N8 * V * H
    rows["fused_lmhead_fwd_dhidden_65536x5120xV"] = {"ms": ms, "algorithmic_flops": fl,
                                                     "achieved_tflops": fl / ms / 1e9,
                                                     "frac": fl / ms / 1e9 / tpeak, "throughput": N8 / (ms / 1e3),
                                                     "unit": "tokens/s", "bound": "tensor"}
    grads8 = lambda: L.leap_fused_lmhead_logprobs(hidden, W, ids8, old8, st8.adv, st8.w, dhidden=dh, want_dW=True,
                                                  dW=dW, workspace=ws8)
    grads8()
    ms = _timed_launches(grads8, 3, stream)
    fl = 8.0 * N8 * V * H
    rows["fused_lmhead_fwd_dhidden_dW_65536x5120xV"] = {"ms": ms, "algorithmic_flops": fl,
                                                        "achieved_tflops": fl / ms / 1e9,
                                                        "frac": fl / ms / 1e9 / tpeak, "throughput": N8 / (ms / 1e3),
                                                        "unit": "tokens/s", "bound": "tensor"}
    # The weight-gradient GEMM alone: dW[V x H] += DL[8,192 x V]^T . hidden[8,192 x H].
    dl8 = synth.normal((8192, V), 1e-3, 505, device, dtype=torch.bfloat16)
    gw = lambda: L.leap_gemm_bf16_tn_f32(dl8, hidden[:8192], out=dW, accumulate=True)
    gw()
    ms = _timed_launches(gw, 5, stream)
    fl = 2.0 * 8192 * V * H
    rows["gemm_bf16_tn_f32_Vx5120x8192"] = {"ms": ms, "algorithmic_flops": fl, "achieved_tflops": fl / ms / 1e9,
                                            "frac": fl / ms / 1e9 / tpeak, "bound": "tensor"}
    del hidden, W, dh, dW, dl8, ws8, flush_buf
    torch.cuda.synchronize()
    return rows


def lmhead_only(args):
    """The fused lm-head alone (H = 5,120, V = 151,936 unless --lmhead-vocab) on
    --lmhead-tokens tokens: --warmup untimed calls, then --steps timed ones;
    prints one JSON line."""
    from paper_2608_01804_gb300 import build
    build.build()
    from paper_2608_01804_gb300 import leap as L
    from paper_2608_01804_gb300 import synth
    device = torch.device("cuda", 0)
    N, H, Vp = args.lmhead_tokens, 5120, args.lmhead_vocab or V
    hidden = synth.normal((N, H), 1.0, 500, device, dtype=torch.bfloat16)
    W = synth.normal((Vp, H), 0.02, 501, device, dtype=torch.bfloat16)
    ids = synth.token_ids(N, Vp, 502, device)
    old = synth.normal(N, 1.0, 503, device) - 12.0
    adv = synth.normal(N, 1.0, 504, device)
    w = torch.full((N,), 1.0 / N, device=device)
    ws = torch.empty(L.leap_fused_lmhead_workspace_size(N, H, Vp, True, args.lmhead_dw), dtype=torch.uint8,
                     device=device)
    dh = torch.empty_like(hidden)
    dW = torch.empty((Vp, H), dtype=torch.float32, device=device) if args.lmhead_dw else None
    run = lambda: L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, dhidden=dh, want_dW=args.lmhead_dw,
                                               dW=dW, workspace=ws)
    for _ in range(args.warmup):
        run()
    ms = _timed_launches(run, args.steps, torch.cuda.current_stream())
    fl = (8.0 if args.lmhead_dw else 6.0) * N * Vp * H
    print(json.dumps({"lmhead_tokens": N, "vocab": Vp, "dW": args.lmhead_dw, "ms": ms, "tflops": fl / ms / 1e9,
                      "frac": fl / ms / 1e9 / measured_tensor_peak()}), flush=True)


def rank_only(args):
    """Rank advantages alone on the tournament workload (65,536 groups x 64
    rollouts, M = 3): --warmup untimed launches, then --steps timed ones,
    each after an L2 flush; prints one JSON line."""
    from paper_2608_01804_gb300 import build
    build.build()
    from paper_2608_01804_gb300 import leap as L
    from paper_2608_01804_gb300 import synth
    device = torch.device("cuda", 0)
    pt, nt, _, _ = synth.tournament_outcomes()
    G, M = 64, 3
    n = pt.size
    pt_d = torch.as_tensor(pt).to(device)
    nt_d = torch.as_tensor(nt).to(device)
    out = L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=50, tau_max=56, gamma=0.9)
    fn = lambda: L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=50, tau_max=56, gamma=0.9, out=out)
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    for _ in range(args.warmup):
        fn()
    ms = _timed_launches(fn, args.steps, torch.cuda.current_stream(), lambda: flush_buf.fill_(1),
                         lead_cycles=LEAD_CYCLES)
    rank_bytes = n * (2 + 1 + 4 + 4 + 4 + 4 + 4 * M + 1) + n // G
    peak, _ = measured_peaks()
    print(json.dumps({"rank_rollouts": n, "ms": ms, "gbs": rank_bytes / ms / 1e6,
                      "frac": rank_bytes / ms / 1e6 / peak}), flush=True)


def tokens_only(args):
    """Per-rollout token counts + per-token scatter alone (the two calls, then
    the one-launch call) on the packed multi-turn batch or, with
    --tokens-layout tiny, the small padded batch: --warmup untimed calls, then
    --steps timed ones, each after an L2 flush; prints one JSON line."""
    from paper_2608_01804_gb300 import build
    build.build()
    from paper_2608_01804_gb300 import leap as L
    from paper_2608_01804_gb300 import synth
    device = torch.device("cuda", 0)
    b = synth.tiny_batch() if args.tokens_layout == "tiny" else synth.multiturn_dcp_batch()
    pt_d = torch.as_tensor(b.pass_turn).to(device)
    nt_d = torch.as_tensor(b.num_turns).to(device)
    tau = (0, b.G) if args.tokens_layout == "tiny" else (8, 15)
    rk = L.leap_group_rank_advantages(pt_d, nt_d, G=b.G, M=b.M, tau_min=tau[0], tau_max=tau[1], gamma=0.9)
    so = torch.as_tensor(b.seg_offsets).to(device)
    sr = torch.as_tensor(b.seg_rollout).to(device)
    st_ = torch.as_tensor(b.seg_turn).to(device)
    Lc, tot = L.leap_rollout_token_counts(b.N, so, sr, st_, rk["T_eff"], M=b.M)
    adv, w = L.leap_scatter_turn_advantages(b.N, so, sr, st_, rk["turn_adv"], rk["T_eff"], Lc, tot, M=b.M)

    def tok():
        L.leap_rollout_token_counts(b.N, so, sr, st_, rk["T_eff"], M=b.M, L=Lc, totals=tot)
        L.leap_scatter_turn_advantages(b.N, so, sr, st_, rk["turn_adv"], rk["T_eff"], Lc, tot, M=b.M, adv=adv, w=w)
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    for _ in range(args.warmup):
        tok()
    ms = _timed_launches(tok, args.steps, torch.cuda.current_stream(), lambda: flush_buf.fill_(1),
                         lead_cycles=LEAD_CYCLES)
    one = lambda: L.leap_token_advantages(b.N, so, sr, st_, rk["turn_adv"], rk["T_eff"], M=b.M, L=Lc, totals=tot,
                                          adv=adv, w=w)
    for _ in range(args.warmup):
        one()
    ms1 = _timed_launches(one, args.steps, torch.cuda.current_stream(), lambda: flush_buf.fill_(1),
                          lead_cycles=LEAD_CYCLES)
    peak, _ = measured_peaks()
    print(json.dumps({"tokens": b.N, "segments": int(b.seg_rollout.size), "ms": ms, "gbs": 8 * b.N / ms / 1e6,
                      "frac": 8 * b.N / ms / 1e6 / peak, "one_launch_ms": ms1,
                      "one_launch_frac": 8 * b.N / ms1 / 1e6 / peak}), flush=True)


def short_rows(args):
    """The fused loss forward + backward (with its two reduction launches) on
    short vocabularies, through the default entry point and with
    LEAP_LOSS_SINGLE_READ: --warmup untimed calls, then --steps timed ones of
    each, each after an L2 flush; one JSON line per (V, rows).  Rows of
    V <= 32,768 take the short-row kernel either way."""
    from paper_2608_01804_gb300 import build
    build.build()
    from paper_2608_01804_gb300 import leap as L
    from paper_2608_01804_gb300 import synth
    device = torch.device("cuda", 0)
    stream = torch.cuda.current_stream()
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    peak, _ = measured_peaks()
    cases = [(1024, 16384), (1024, 262144), (1000, 262144), (4096, 65536), (8192, 32768), (16384, 16384), (32000, 8192),
             (32768, 8192), (65536, 4096)]
    if args.short_case:
        cases = [tuple(int(x) for x in args.short_case.split("x"))]
    for Vs, N in cases:
        z = synth.logits(N, Vs, 2.0, 1, device, ld=(Vs + 7) // 8 * 8)
        ids = synth.token_ids(N, Vs, 2, device)
        old = torch.full((N,), -7.0, device=device)
        adv = synth.normal(N, 1.0, 3, device)
        w = torch.full((N,), 1.0 / N, device=device)
        dl = torch.empty_like(z)
        ws = L.loss_workspace(N, Vs, device)
        loss = torch.zeros(1, device=device)
        line = {"V": Vs, "rows": N, "algorithmic_bytes": 4 * Vs * N}
        for name, sr in (("default", False), ("single_read", True)):
            fn = lambda sr=sr: L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=Vs, loss=loss, dlogits=dl,
                                                    want_outputs=False, workspace=ws, single_read=sr)
            for _ in range(max(1, args.warmup)):
                fn()
            ms = _timed_launches(fn, args.steps, stream, lambda: flush_buf.fill_(1), lead_cycles=LEAD_CYCLES)
            line[name + "_us"] = ms * 1e3
            line[name + "_frac"] = 4 * Vs * N / ms / 1e6 / peak
        print(json.dumps(line), flush=True)
        del z, dl, ws


def logprobs_only(args):
    """Token log-probs and the forward-only loss alone on the single-turn batch
    (32,768 x 151,936): --warmup untimed calls, then --steps timed ones of
    each; prints one JSON line."""
    from paper_2608_01804_gb300 import build
    build.build()
    from paper_2608_01804_gb300 import leap as L
    from paper_2608_01804_gb300.step import GrpoStep
    device = torch.device("cuda", 0)
    batch, logits, ids, old = make_inputs(0, device)
    step = GrpoStep(batch, V, device, gamma=1.0, tau=(0, batch.G), use_gate_in=False)
    step.advantages()
    N = logits.shape[0]
    live = int((step.w != 0).sum().item())
    logp = torch.empty(N, dtype=torch.float32, device=device)
    lse = torch.empty(N, dtype=torch.float32, device=device)
    ws = L.loss_workspace(N, V, device)
    lp = lambda: L.leap_token_logprobs(logits, ids, V=V, logp=logp, lse=lse)
    fwd = lambda: L.leap_grpo_loss_fwd(logits, ids, old, step.adv, step.w, V=V, loss=step.loss, lse=lse,
                                       want_dlogits=False, want_outputs=False, workspace=ws)
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        lp()
        fwd()
    ms_lp = _timed_launches(lp, args.steps, stream)
    ms_f = _timed_launches(fwd, args.steps, stream)
    peak, _ = measured_peaks()
    b_lp, b_f = 2 * V * N + 12 * N, 2 * V * live + 16 * N
    print(json.dumps({"logprobs_ms": ms_lp, "logprobs_frac": b_lp / ms_lp / 1e6 / peak,
                      "fwd_ms": ms_f, "fwd_frac": b_f / ms_f / 1e6 / peak}), flush=True)


def main():
    args = parse_args()
    if args.oracle_config_one:
        print(json.dumps(_oracle_one(args.oracle_config_one, args.cpu_seconds)), flush=True)
        return
    if args.oracle_configs:
        oracle_configs(args)
        return
    if args.impl == "reference":
        reference_arm(args)
        return
    if args.lmhead_tokens:
        lmhead_only(args)
        return
    if args.rank_only:
        rank_only(args)
        return
    if args.tokens_only:
        tokens_only(args)
        return
    if args.logprobs_only:
        logprobs_only(args)
        return
    if args.short_rows:
        short_rows(args)
        return
    if args.multiturn:
        from paper_2608_01804_gb300 import build
        build.build()
        torch.cuda.set_device(0)
        peak, _ = measured_peaks()
        print(json.dumps(multiturn_step(torch.device("cuda", 0), peak, steps=args.steps, warmup=args.warmup)),
              flush=True)
        return
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    pg = None
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=device)
        pg = torch.distributed.group.WORLD

    from paper_2608_01804_gb300 import build
    build.build()
    from paper_2608_01804_gb300.step import GrpoStep

    batch, logits, ids, old = make_inputs(rank, device, args.prompts)
    N = batch.N
    n_valid = valid_tokens(batch)
    step = GrpoStep(batch, V, device, gamma=1.0, tau=(0, batch.G), use_gate_in=False)
    dlogits = torch.empty_like(logits)
    stream = torch.cuda.current_stream()

    def barrier():
        if pg is not None:
            torch.distributed.barrier()

    from paper_2608_01804_gb300 import leap as L
    L.leap_get_device_status()
    for _ in range(max(3, args.warmup)):
        step.run(logits, ids, old, dlogits, pg)
    torch.cuda.synchronize()
    flags = L.leap_get_device_status()
    if flags:
        raise RuntimeError("libleap device status 0x%x after the warm-up steps" % flags)
    live_rows = int((step.w != 0).sum().item())
    assert live_rows == n_valid

    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    clocks = clock_sampler(device)
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_stop = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(K):
        step.advantages(pg)
        ev[k][0].record(stream)
        step.loss_pass(logits, ids, old, dlogits)
        ev[k][1].record(stream)
    t_stop.record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    elapsed_ms = t_start.elapsed_time(t_stop)
    launch_times = sorted(a.elapsed_time(b) for a, b in ev)
    loss_ms = sum(launch_times) / K
    if pg is not None:
        t = torch.tensor([elapsed_ms], device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        elapsed_ms = float(t.item())
    ms_per_step = elapsed_ms / K
    value = n_valid * world / (ms_per_step / 1e3)

    peak, peak_kind = measured_peaks()
    alg_bytes = live_rows * 4 * V + (N - live_rows) * 2 * V + 16 * N
    achieved = alg_bytes / (loss_ms / 1e3) / 1e9
    traffic = None
    if KNOWN_TRAFFIC and KNOWN_TRAFFIC.get("src_sha256") == _src_sha():
        traffic = KNOWN_TRAFFIC["bytes_per_launch"]
    spread = {"median_ms": launch_times[K // 2], "min_ms": launch_times[0], "max_ms": launch_times[-1],
              "frac_at_median": alg_bytes / (launch_times[K // 2] / 1e3) / 1e9 / peak,
              "frac_of_nominal_7900_gbs": achieved / 7900.0}
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "launch_spread": spread,
                "traffic": traffic, "kernel": "fused_loss_pipe_kernel<4,8,3,11,1024> persistent, rows pipelined (+2 reduce launches in the timing)",
                "algorithmic_bytes_per_launch": alg_bytes, "launch_ms": loss_ms, "peak_source": peak_kind}

    # End to end through the same public calls, inputs copied from pinned host memory every step.
    e2e = None
    if not args.no_e2e:
        host = {k: t.cpu().pin_memory() for k, t in dict(logits=logits, ids=ids, old=old,
                                                         pass_turn=step.pass_turn, num_turns=step.num_turns,
                                                         seg_offsets=step.seg_offsets, seg_rollout=step.seg_rollout,
                                                         seg_turn=step.seg_turn).items()}
        dev = dict(logits=logits, ids=ids, old=old, pass_turn=step.pass_turn, num_turns=step.num_turns,
                   seg_offsets=step.seg_offsets, seg_rollout=step.seg_rollout, seg_turn=step.seg_turn)
        small_h2d = sum(t.numel() * t.element_size() for k, t in host.items() if k != "logits")
        loss_host = torch.empty(1, dtype=torch.float32).pin_memory()
        E = max(1, args.e2e_steps)

        def e2e_step():
            for k, t in host.items():      # the small inputs; the logits stream in run_streamed
                if k != "logits":
                    dev[k].copy_(t, non_blocking=True)
            step.run_streamed(host["logits"], dev["ids"], dev["old"], dlogits, chunk_rows=E2E_CHUNK_ROWS, pg=pg)
            loss_host.copy_(step.loss, non_blocking=True)

        e2e_step()
        torch.cuda.synchronize()
        barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(E):
            e2e_step()
        b.record(stream)
        torch.cuda.synchronize()
        e_ms = a.elapsed_time(b) / E
        if pg is not None:
            t = torch.tensor([e_ms], device=device)
            torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
            e_ms = float(t.item())
        # run_streamed copies only the logit rows that can carry loss weight (generated turns; the loss
        # never reads a padding row's logits and writes its dlogits as zeros): the bytes it counted.
        h2d = small_h2d + step.h2d_logit_bytes
        e2e = {"value": n_valid * world / (e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": 4, "ms_per_step": e_ms, "steps": E,
               "h2d_logit_rows_per_step": step.h2d_logit_bytes // (logits.shape[1] * logits.element_size()),
               "note": "logits of rows that cannot carry loss weight (padding) stay on the host"}
        del host

    rows = None
    if rank == 0 and not args.no_rows and args.prompts == 16:
        rows = measure_rows(device, logits, ids, old, step, peak)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rate1, n_rows, valid1, secs1 = cpu_oracle_rate(batch, logits, ids, old, args.cpu_seconds)
        rate, workers, valid, secs = cpu_oracle_rate_all_cores(batch, logits, ids, old)
        cpu = {"value": rate, "unit": UNIT, "cores": workers, "kind": "oracle",
               "sample": "the whole batch (%d valid tokens): rank/token oracle once, then loss fwd and dlogits of "
                         "every row in 32-row blocks over %d spawned worker processes, %.1f s wall"
                         % (valid, workers, secs),
               "cpu_model": _cpu_model(),
               "single_thread": {"value": rate1, "cores": 1,
                                 "sample": "rank/token oracle on the whole batch + loss fwd and dlogits on the first "
                                           "%d rows (%d valid tokens), %.1f s of CPU time" % (n_rows, valid1, secs1)}}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": args.warmup,
                "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "data": "synthetic",
                "config": workload_config(args.prompts, N, n_valid, world),
                "roofline": roofline, "rows": rows, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": K * step.launches_per_run(pg), "clocks": clk}
        print(json.dumps(line), flush=True)
    if pg is not None:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
