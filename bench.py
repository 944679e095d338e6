"""Benchmark of the SONIC Nexus-KV attention path on GB300.

One step = one mixed serving step over 28 layers (28 query / 4 KV heads,
D = 128, bf16), the whole hot path in order:
  1. compaction: the 8 sequences that resume with a new turn drop the bodies
     of their raw histories (~U[4k, 64k] tokens each) -- retention rule;
  2. masked prefill: their new turns (~U[256, 2048] tokens) attend over the
     retained cache plus themselves under the Sec. 3.2 mask;
  3. decode: the other 56 sequences decode one token over retained caches of
     ~1k-18k rows.
All three calls go through the C ABI on one CUDA stream.

Reported:
  value        prefill TFLOP/s (algorithmic: 4 * D * Hq * visible pairs) over
               the prefill launches of the timed steps (the dominant kernel);
  decode       HBM GB/s (retained K/V read + q/O) over the decode launches;
  compaction   HBM GB/s (kept rows read + written) over the compaction launches;
  e2e          the same metric with every step's inputs copied from pinned
               host memory and its outputs read back inside the timed region;
  roofline     the prefill kernel against the measured bf16 peak;
  cpu_baseline the double-precision oracle timed on a bounded sample.
`--impl reference` times the oracle itself on that sample (reference arm).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "Nexus-KV attn: decode HBM GB/s & prefill TFLOP/s vs GB300 peak"
WORKLOAD = ("mixed serving step: 64 ragged sequences, 28 layers, 28/4 heads, D=128, bf16; "
            "8 compact a 4k-64k raw history then prefill a 256-2048-token turn, 56 decode "
            "over 1k-18k retained rows")


def max_over_ranks(values, device="cpu"):
    """Element-wise maximum of `values` over all ranks (the timing rule: the
    slowest rank defines the step); identity on a single process."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def weak_rate(work_per_step: float, steps: int, world: int, ms: float, scale: float) -> float:
    """Whole-job throughput of N replicas: every rank processes the same work
    per step, the job time is the slowest rank's."""
    return work_per_step * steps * world / (ms * 1e-3) / scale


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"],
                    bf16_sus=d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


# ---------------------------------------------------------------------------
# Workload (host side: layout bookkeeping only)
# ---------------------------------------------------------------------------

class Layout:
    def __init__(self, seed: int = 1, n_layers: int = 0):
        from paper_2601_21927_gb300 import inputs
        self.ms = ms = inputs.mixed_serving(seed=seed)
        h = ms.heads
        self.NL, self.HQ, self.HKV, self.D = h.n_layers, h.hq, h.hkv, h.d
        if n_layers > 0:
            self.NL = n_layers
        self.row_bytes = self.HKV * self.D * 2
        # raw histories of the prefill sequences (packed)
        self.raw = inputs.Batch(ms.raw_hist)
        self.n_pre = len(ms.raw_hist)
        self.q_len = np.array(ms.prefill_q, np.int32)
        self.ret_pre = np.array([d.recipe_retained for d in ms.raw_hist], np.int32)
        # retained-cache buffer: decode sequences first, then the prefill region
        self.dec_len = np.array([d.recipe_retained + 1 for d in ms.decode_hist], np.int32)
        self.n_dec = len(self.dec_len)
        self.dec_start = np.concatenate([[0], np.cumsum(self.dec_len)[:-1]]).astype(np.int32)
        self.T_dec = int(self.dec_len.sum())
        self.pre_off = np.concatenate([[0], np.cumsum(self.ret_pre + self.q_len)[:-1]]).astype(np.int32)
        self.T_pre = int((self.ret_pre + self.q_len).sum())
        self.T_ret = self.T_dec + self.T_pre
        self.k_start_pre = (self.T_dec + self.pre_off).astype(np.int32)
        self.k_len_pre = (self.ret_pre + self.q_len).astype(np.int32)
        self.q_start = np.concatenate([[0], np.cumsum(self.q_len)[:-1]]).astype(np.int32)
        self.T_q = int(self.q_len.sum())
        # role / segment numbers of every row of the retained buffer
        role = np.zeros(self.T_ret, np.uint8)
        seg = np.zeros(self.T_ret, np.int32)
        for b, d in enumerate(ms.decode_hist):
            r, s = d.retained_arrays()
            s0 = self.dec_start[b]
            role[s0:s0 + len(r)] = r
            seg[s0:s0 + len(r)] = s
            role[s0 + len(r)] = 3
            seg[s0 + len(r)] = len(d.segments) + 1
        for b, d in enumerate(ms.raw_hist):
            r, s = d.retained_arrays()
            s0 = self.k_start_pre[b]
            role[s0:s0 + len(r)] = r
            seg[s0:s0 + len(r)] = s
            role[s0 + len(r):s0 + len(r) + self.q_len[b]] = 3
            seg[s0 + len(r):s0 + len(r) + self.q_len[b]] = len(d.segments) + 1
        self.role_ret, self.seg_ret = role, seg

    # algorithmic work per step
    def prefill_flops(self) -> float:
        pairs = sum(int(q) * int(r) + int(q) * (int(q) + 1) // 2
                    for q, r in zip(self.q_len, self.ret_pre))
        return 4.0 * self.D * self.HQ * pairs * self.NL

    def decode_bytes(self) -> float:
        kv = float(self.dec_len.sum()) * self.row_bytes * 2
        qo = 2.0 * self.n_dec * self.HQ * self.D * 2
        meta = self.n_dec * 8.0
        return (kv + qo + meta) * self.NL

    def compact_bytes(self) -> float:
        return float(self.ret_pre.sum()) * self.row_bytes * 2 * 2 * self.NL


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

class GpuStep:
    def __init__(self, lay: Layout, device, seed: int = 0):
        import torch
        from paper_2601_21927_gb300 import inputs, sonic
        self.torch, self.sonic, self.lay = torch, sonic, lay
        t = lambda a: torch.as_tensor(a).to(device)
        NL, HQ, HKV, D = lay.NL, lay.HQ, lay.HKV, lay.D
        bf = torch.bfloat16
        # KV cache state (resident)
        self.rawK = inputs.randn((NL, lay.raw.total, HKV, D), seed=seed + 1, device=device)
        self.rawV = inputs.randn((NL, lay.raw.total, HKV, D), seed=seed + 2, device=device)
        self.Kret = inputs.randn((NL, lay.T_ret, HKV, D), seed=seed + 3, device=device)
        self.Vret = inputs.randn((NL, lay.T_ret, HKV, D), seed=seed + 4, device=device)
        self.raw_role, self.raw_seg = t(lay.raw.role), t(lay.raw.seg)
        self.raw_kstart, self.raw_klen = t(lay.raw.k_start), t(lay.raw.k_len)
        self.reserve = t(lay.q_len)
        self.offsets = torch.zeros(lay.n_pre + 1, dtype=torch.int32, device=device)
        self.role_ret, self.seg_ret = t(lay.role_ret), t(lay.seg_ret)
        self.k_start_pre, self.k_len_pre = t(lay.k_start_pre), t(lay.k_len_pre)
        self.q_start, self.q_len = t(lay.q_start), t(lay.q_len)
        self.dec_start, self.dec_len = t(lay.dec_start), t(lay.dec_len)
        # per-step inputs and outputs
        self.Qp = inputs.randn((NL, lay.T_q, HQ, D), seed=seed + 5, device=device)
        self.Op = torch.empty_like(self.Qp)
        self.qd = inputs.randn((NL, lay.n_dec, HQ, D), seed=seed + 6, device=device)
        self.Od = torch.empty_like(self.qd)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        self.outK = self.Kret[:, lay.T_dec:]
        self.outV = self.Vret[:, lay.T_dec:]
        # workspaces (caller-owned; sized once)
        self.ws_c = self.ws_p = self.ws_d = None
        self.launches_per_step = 4 + 2 + 2

    def compact(self, stream=None):
        self.ws_c = self.sonic.sonic_compact_kv(
            self.rawK, self.rawV, self.raw_seg, self.raw_role, self.outK, self.outV,
            self.offsets, k_start=self.raw_kstart, k_len=self.raw_klen, reserve=self.reserve,
            status=self.status, workspace=self.ws_c, stream=stream)

    def prefill(self, stream=None):
        lay = self.lay
        self.ws_p = self.sonic.sonic_attn_prefill(
            self.Qp, self.Kret, self.Vret, self.seg_ret, self.role_ret, self.Op,
            k_start=self.k_start_pre, k_len=self.k_len_pre, q_start=self.q_start,
            q_len=self.q_len, max_q_len=int(lay.q_len.max()), max_k_len=int(lay.k_len_pre.max()),
            status=self.status, workspace=self.ws_p, stream=stream)

    def decode(self, stream=None):
        self.ws_d = self.sonic.sonic_attn_decode(
            self.qd, self.Kret, self.Vret, self.dec_len, self.Od, kv_start=self.dec_start,
            max_len=int(self.lay.dec_len.max()), status=self.status, workspace=self.ws_d,
            stream=stream)

    def step(self, stream=None):
        self.compact(stream)
        self.prefill(stream)
        self.decode(stream)


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.file = None

    def start(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [l.strip().split(", ") for l in self.file.read().splitlines() if l.strip()]
        os.unlink(self.file.name)
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx = max(mx, float(r[2]))
                for n, v in zip(names, r[5:9]):
                    if v.strip() == "Active":
                        reasons.add(n)
            except (ValueError, IndexError):
                continue
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def run_gpu(args, rank: int, world: int):
    import torch
    import torch.distributed as dist
    from paper_2601_21927_gb300 import sonic

    local = int(os.environ.get("LOCAL_RANK", "0"))
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    sonic.load()
    lay = Layout(n_layers=args.layers)
    g = GpuStep(lay, device, seed=17 * rank)
    stream = torch.cuda.Stream(device)
    torch.cuda.synchronize()
    if args.only:
        # one phase alone (small captures for the profiler)
        fn = {"compact": g.compact, "prefill": g.prefill, "decode": g.decode}[args.only]
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                fn(stream)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(args.steps):
                fn(stream)
            b.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / max(args.steps, 1)
        work = {"compact": lay.compact_bytes(), "prefill": lay.prefill_flops(),
                "decode": lay.decode_bytes()}[args.only]
        rate = work / (ms * 1e-3) / (1e12 if args.only == "prefill" else 1e9)
        return {"only": args.only, "n_layers": lay.NL, "ms_per_launch": round(ms, 4),
                "rate": round(rate, 2), "unit": "TFLOP/s" if args.only == "prefill" else "GB/s",
                "status": sonic.read_status(g.status)}, lay

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    ev = lambda: torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g.step(stream)
    torch.cuda.synchronize()
    if sonic.read_status(g.status) != 0:
        raise RuntimeError(f"device status {sonic.read_status(g.status)} after warm-up")

    marks = [(ev(), ev(), ev(), ev()) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier()
    clocks.start()
    t_start, t_end = ev(), ev()
    with torch.cuda.stream(stream):
        t_start.record(stream)
        for e0, e1, e2, e3 in marks:
            e0.record(stream)
            g.compact(stream)
            e1.record(stream)
            g.prefill(stream)
            e2.record(stream)
            g.decode(stream)
            e3.record(stream)
        t_end.record(stream)
    barrier()
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_end)
    c_ms = sum(a.elapsed_time(b) for a, b, _, _ in marks)
    p_ms = sum(b.elapsed_time(c) for _, b, c, _ in marks)
    d_ms = sum(c.elapsed_time(d) for _, _, c, d in marks)
    if sonic.read_status(g.status) != 0:
        raise RuntimeError("device status set during the timed steps")

    # ---------------- end to end: host buffers through the public calls
    # Every step copies its inputs from pinned host memory (new-turn Q, decode
    # q, the new tokens' K/V rows) and reads its outputs back (prefill O,
    # decode O).  Steps are pipelined over a compute stream and a copy stream,
    # as a server would run them: outputs of step k-1 and then inputs of step
    # k+1 move while step k computes (Q/O double-buffered); the K/V rows land in
    # one contiguous copy and are appended into their cache rows by indexed
    # device copies just before the step that reads them.
    pin = lambda t: t.cpu().pin_memory()
    hQ, hqd = pin(g.Qp), pin(g.qd)
    hOp, hOd = torch.empty_like(hQ).pin_memory(), torch.empty_like(hqd).pin_memory()
    newK = pin(g.Kret[:, lay.T_dec:][:, 0:1].expand(-1, lay.T_q, -1, -1).contiguous())
    newV = pin(newK.clone())
    dec_rows = lay.dec_start + lay.dec_len - 1
    hdecK = pin(g.Kret[:, torch.as_tensor(dec_rows, device=device).long()])
    hdecV = pin(hdecK.clone())
    stK, stV = torch.empty_like(newK, device=device), torch.empty_like(newV, device=device)
    stdK, stdV = torch.empty_like(hdecK, device=device), torch.empty_like(hdecV, device=device)
    sets = [(g.Qp, g.qd, g.Op, g.Od),
            (torch.empty_like(g.Qp), torch.empty_like(g.qd), torch.empty_like(g.Op),
             torch.empty_like(g.Od))]
    h2d = (hQ.numel() + hqd.numel() + newK.numel() + newV.numel() + hdecK.numel() +
           hdecV.numel()) * 2
    d2h = (hOp.numel() + hOd.numel()) * 2
    s_io = torch.cuda.Stream(device)

    # cache rows the new tokens go to (indexed copies on the compute stream)
    pre_rows = torch.as_tensor(np.concatenate(
        [np.arange(lay.k_start_pre[b] + lay.ret_pre[b],
                   lay.k_start_pre[b] + lay.ret_pre[b] + lay.q_len[b])
         for b in range(lay.n_pre)]), device=device).long()
    dec_rows_t = torch.as_tensor(dec_rows, device=device).long()

    def append_rows():
        g.Kret.index_copy_(1, pre_rows, stK)
        g.Vret.index_copy_(1, pre_rows, stV)
        g.Kret.index_copy_(1, dec_rows_t, stdK)
        g.Vret.index_copy_(1, dec_rows_t, stdV)

    def e2e_run(nsteps):
        # One copy stream carries both directions, one after the other: on this
        # host link concurrent host->device and device->host copies slow each
        # other down far more than running them back to back.  Per step k it
        # reads back step k-1's outputs, then writes step k+1's inputs.
        ev_in = [ev() for _ in range(nsteps)]
        ev_app = [ev() for _ in range(nsteps)]
        ev_comp = [ev() for _ in range(nsteps)]
        ev_out = [ev() for _ in range(nsteps)]
        start, end = ev(), ev()
        start.record(stream)
        s_io.wait_event(start)

        def inputs_in(k):
            Qp, qd = sets[k % 2][0], sets[k % 2][1]
            with torch.cuda.stream(s_io):
                if k >= 2:
                    s_io.wait_event(ev_comp[k - 2])  # set k%2 no longer read
                if k >= 1:
                    s_io.wait_event(ev_app[k - 1])   # staging buffers consumed
                Qp.copy_(hQ, non_blocking=True)
                qd.copy_(hqd, non_blocking=True)
                stK.copy_(newK, non_blocking=True)
                stV.copy_(newV, non_blocking=True)
                stdK.copy_(hdecK, non_blocking=True)
                stdV.copy_(hdecV, non_blocking=True)
                ev_in[k].record(s_io)

        def outputs_out(k):
            Op, Od = sets[k % 2][2], sets[k % 2][3]
            with torch.cuda.stream(s_io):
                s_io.wait_event(ev_comp[k])
                hOp.copy_(Op, non_blocking=True)
                hOd.copy_(Od, non_blocking=True)
                ev_out[k].record(s_io)

        inputs_in(0)
        for k in range(nsteps):
            Qp, qd, Op, Od = sets[k % 2]
            with torch.cuda.stream(stream):
                stream.wait_event(ev_in[k])
                if k >= 2:
                    stream.wait_event(ev_out[k - 2])  # O of set k%2 read back
                append_rows()
                ev_app[k].record(stream)
                g.Qp, g.qd, g.Op, g.Od = Qp, qd, Op, Od
                g.step(stream)
                ev_comp[k].record(stream)
            if k >= 1:
                outputs_out(k - 1)
            if k + 1 < nsteps:
                inputs_in(k + 1)
        outputs_out(nsteps - 1)
        end.record(s_io)
        return start, end

    e2e_run(max(2, args.warmup // 2))
    barrier()
    e0, e1 = e2e_run(args.steps)
    barrier()
    e2e_ms = e0.elapsed_time(e1)
    g.Qp, g.qd, g.Op, g.Od = sets[0]

    # max over ranks
    total_ms, c_ms, p_ms, d_ms, e2e_ms = max_over_ranks([total_ms, c_ms, p_ms, d_ms, e2e_ms],
                                                        device)
    K = args.steps
    pk = _peaks()
    pf = lay.prefill_flops()
    value = weak_rate(pf, K, world, p_ms, 1e12)
    dec_gbs = weak_rate(lay.decode_bytes(), K, world, d_ms, 1e9)
    cmp_gbs = weak_rate(lay.compact_bytes(), K, world, c_ms, 1e9)
    e2e_val = weak_rate(pf, K, world, e2e_ms, 1e12)
    prof = _traffic()
    achieved = pf / (p_ms / K * 1e-3) / 1e12
    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world,
        "steps": K, "warmup": args.warmup, "ms_per_step": round(total_ms / K, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) K/V/Q; dialogue shapes drawn from the workload recipe)",
        "config": {"workload": WORKLOAD, "n_layers": lay.NL, "heads_q": lay.HQ,
                   "heads_kv": lay.HKV, "head_dim": lay.D, "prefill_seqs": lay.n_pre,
                   "prefill_query_rows": lay.T_q, "decode_seqs": lay.n_dec,
                   "decode_retained_rows": int(lay.dec_len.sum()),
                   "raw_history_rows": lay.raw.total, "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (decode reads %.1f GB/step)" % (
                       lay.decode_bytes() / 1e9),
                   "value_basis": "prefill flops / prefill launch time"},
        "decode": {"value": round(dec_gbs, 1), "unit": "GB/s",
                   "ms_per_step": round(d_ms / K, 3),
                   "roofline": {"bound": "hbm", "achieved": round(dec_gbs / world, 1),
                                "peak": pk["hbm"], "unit": "GB/s",
                                "frac": round(dec_gbs / world / pk["hbm"], 4),
                                "traffic": prof.get("decode")}},
        "compaction": {"value": round(cmp_gbs, 1), "unit": "GB/s",
                       "ms_per_step": round(c_ms / K, 3),
                       "roofline": {"bound": "hbm", "achieved": round(cmp_gbs / world, 1),
                                    "peak": pk["hbm"], "unit": "GB/s",
                                    "frac": round(cmp_gbs / world / pk["hbm"], 4),
                                    "traffic": prof.get("compact")}},
        "prefill_ms_per_step": round(p_ms / K, 3),
        "roofline": {"bound": "tensor", "achieved": round(achieved, 2),
                     "peak": pk["bf16"], "unit": "TFLOP/s",
                     "frac": round(achieved / pk["bf16"], 4), "traffic": prof.get("prefill"),
                     "peak_source": pk["source"] + " bf16 burst (the kernel runs at the maximum "
                                                   "SM clock; see clocks)",
                     "peak_sustained": pk["bf16_sus"],
                     "frac_of_sustained": round(achieved / pk["bf16_sus"], 4)},
        "e2e": {"value": round(e2e_val, 2), "unit": "TFLOP/s",
                "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                "ms_per_step": round(e2e_ms / K, 3)},
        "gpu_launches": g.launches_per_step * K,
        "clocks": clk,
    }
    return out, lay


def _traffic():
    """DRAM bytes per launch from the committed ncu summary (if it matches)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return {}
    with open(p) as f:
        return json.load(f)


# ---------------------------------------------------------------------------
# Oracle arm (CPU)
# ---------------------------------------------------------------------------

def oracle_sample(lay: Layout, n_rows: int = 512, threads: int = None):
    """Time the oracle on a bounded sample of the step's prefill: n_rows query
    rows of every prefill sequence (spread over the turn), all 28 heads,
    layer 0.  Returns (TFLOP/s, seconds, cores, description)."""
    import oracle
    from concurrent.futures import ThreadPoolExecutor
    rng = np.random.default_rng(5)
    orc = oracle.default()
    threads = threads or os.cpu_count() or 1
    jobs = []
    flops = 0.0
    for b in range(lay.n_pre):
        R = int(lay.ret_pre[b])
        L = R + int(lay.q_len[b])
        K = rng.standard_normal((L, lay.HKV, lay.D))
        V = rng.standard_normal((L, lay.HKV, lay.D))
        role = lay.role_ret[lay.k_start_pre[b]:lay.k_start_pre[b] + L]
        seg = lay.seg_ret[lay.k_start_pre[b]:lay.k_start_pre[b] + L]
        rows = np.linspace(R, L - 1, n_rows).astype(np.int64)
        for r in rows:
            Q = rng.standard_normal((1, lay.HQ, lay.D))
            jobs.append((Q, K, V, role, seg, np.array([r])))
            flops += 4.0 * lay.D * lay.HQ * (r + 1)
    t0 = time.perf_counter()
    with ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(lambda j: orc.attn_masked(*j), jobs))
    dt = time.perf_counter() - t0
    desc = (f"oracle masked attention, {len(jobs)} query rows ({n_rows} per prefill sequence) "
            f"x {lay.HQ} heads, layer 0, float64, {threads} threads")
    return flops / dt / 1e12, dt, threads, desc


def oracle_decode_sample(lay: Layout, n_layers: int = 4, threads: int = None):
    """Time the oracle's decode on a bounded sample of the step's decode: all
    56 decoding sequences over their retained rows, all 28 query heads, four
    layers.  Returns (GB/s of algorithmic bytes, seconds, cores, description)."""
    import oracle
    from concurrent.futures import ThreadPoolExecutor
    rng = np.random.default_rng(6)
    orc = oracle.default()
    threads = threads or os.cpu_count() or 1
    jobs, by = [], 0.0
    # one buffer of the longest cache; every sequence reads a prefix of it
    n_max = int(lay.dec_len.max())
    Kall = rng.standard_normal((n_max, lay.HKV, lay.D))
    Vall = rng.standard_normal((n_max, lay.HKV, lay.D))
    for _ in range(n_layers):
        for b in range(lay.n_dec):
            n = int(lay.dec_len[b])
            q = rng.standard_normal((lay.HQ, lay.D))
            jobs.append((q, Kall[:n], Vall[:n]))
            by += n * lay.row_bytes * 2 + 2 * lay.HQ * lay.D * 2 + 8
    t0 = time.perf_counter()
    with ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(lambda j: orc.decode(*j), jobs))
    dt = time.perf_counter() - t0
    desc = (f"oracle decode, {lay.n_dec} sequences x {lay.HQ} heads over their retained rows "
            f"({int(lay.dec_len.sum())} rows), {n_layers} layer(s), float64, {threads} threads; "
            f"bf16 bytes the GPU would read")
    return by / dt / 1e9, dt, threads, desc


def oracle_compact_sample(lay: Layout, n_layers: int = 28):
    """Time the oracle's retention rule and row copy on a bounded sample of the
    step's compaction: the 8 raw histories, K and V of n_layers layers.
    Returns (GB/s of algorithmic bytes, seconds, cores, description)."""
    import oracle
    orc = oracle.default()
    rng = np.random.default_rng(7)
    raw = rng.integers(0, 256, size=(1, lay.raw.total, lay.row_bytes), dtype=np.uint8)
    t0 = time.perf_counter()
    for _ in range(n_layers * 2):   # K and V of every layer
        off, ret_len, src = orc.retain(lay.raw.k_start, lay.raw.k_len, lay.raw.role, lay.q_len)
        orc.compact_copy(raw, off, ret_len, src, int(off[-1]))
    dt = time.perf_counter() - t0
    by = float(lay.ret_pre.sum()) * lay.row_bytes * 2 * 2 * n_layers
    desc = (f"oracle retention rule + row copy, {lay.n_pre} raw histories ({lay.raw.total} rows, "
            f"{lay.row_bytes}-byte rows), K and V of {n_layers} layers, 1 thread")
    return by / dt / 1e9, dt, 1, desc


# ---------------------------------------------------------------------------
# Further workloads (`--extra NAME`): one JSON line each, outside the
# benchmark contract line.  Every rate counts algorithmic work only.
# ---------------------------------------------------------------------------

def _ev_time(fn, reps=5, warm=2):
    import torch
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        fn()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def _visible_pairs(role, seg, rows, mode):
    """Visible (query, key) pairs of the Sec. 3.2 mask for query positions
    `rows` of one sequence (host bookkeeping for the flop count)."""
    pos = np.arange(len(role))
    n = 0
    for p in rows:
        body = role == 1
        nex = (role[p] == 2) & (role == 2)
        nexv = True if mode == 0 else (seg <= seg[p])
        v = np.where(body, (seg == seg[p]) & (pos <= p), np.where(nex, nexv, pos <= p))
        n += int(v.sum())
    return n


def extra_masked_prefill():
    """Masked prefill of a whole S_aug (Sec. 3.2): batch 8, 512 system tokens,
    16 segments of 256 body + 32 Nexus tokens, a 512-token current turn (L =
    5632), 32/8 heads, D = 128, one layer; every row a query, both key orders
    and both Nexus readings; then the current turn's rows alone."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    batch, hd = inputs.masked_prefill()
    d = batch.dialogues[0]
    role, seg = d.arrays()
    L = d.length
    t = lambda a: torch.as_tensor(np.asarray(a)).to(dev)
    K = inputs.randn((1, batch.total, hd.hkv, hd.d), seed=1, device=dev)
    V = inputs.randn((1, batch.total, hd.hkv, hd.d), seed=2, device=dev)
    Q = inputs.randn((1, batch.total, hd.hq, hd.d), seed=3, device=dev)
    O = torch.empty_like(Q)
    r_, s_, ks, kl = t(batch.role), t(batch.seg), t(batch.k_start), t(batch.k_len)
    res = {}
    for mode in (0, 1):
        flops = 4.0 * hd.d * hd.hq * _visible_pairs(role, seg, range(L), mode) * batch.B
        for order, oname in ((0, "as_given"), (1, "retained_first")):
            call = lambda ws=None: sonic.sonic_attn_prefill(
                Q, K, V, s_, r_, O, k_start=ks, k_len=kl, q_start=ks, q_len=kl, max_q_len=L,
                max_k_len=L, nexus_vis=mode, key_order=order, workspace=ws)
            ws = call()
            ms = _ev_time(lambda: call(ws))
            res[f"all_rows_{'full' if mode == 0 else 'causal_segments'}_{oname}"] = {
                "ms": round(ms, 3), "tflops": round(flops / ms / 1e9, 1)}
    ql = np.full(batch.B, d.curr_len, np.int32)
    qs = np.concatenate([[0], np.cumsum(ql)[:-1]]).astype(np.int32)
    Qc = inputs.randn((1, int(ql.sum()), hd.hq, hd.d), seed=4, device=dev)
    Oc = torch.empty_like(Qc)
    flops = 4.0 * hd.d * hd.hq * _visible_pairs(role, seg, range(L - d.curr_len, L), 0) * batch.B
    qst, qlt = t(qs), t(ql)
    for order, oname in ((0, "as_given"), (1, "retained_first")):
        call = lambda ws=None: sonic.sonic_attn_prefill(
            Qc, K, V, s_, r_, Oc, k_start=ks, k_len=kl, q_start=qst, q_len=qlt,
            max_q_len=int(ql.max()), max_k_len=L, key_order=order, workspace=ws)
        ws = call()
        ms = _ev_time(lambda: call(ws))
        res[f"current_rows_{oname}"] = {"ms": round(ms, 3), "tflops": round(flops / ms / 1e9, 1)}
    return {"workload": "masked prefill, batch 8 x 5632 rows, 32/8 heads, D=128, 1 layer",
            "results": res}


def extra_prefill_d64():
    """The masked-prefill workload (batch 8 x 5632 rows, every row a query, full
    mask, retained-first key order; and the current-turn rows alone) at
    head_dim 64 with 32/8 heads, beside head_dim 128."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    batch, _ = inputs.masked_prefill()
    d = batch.dialogues[0]
    role, seg = d.arrays()
    L = d.length
    t = lambda a: torch.as_tensor(np.asarray(a)).to(dev)
    r_, s_, ks, kl = t(batch.role), t(batch.seg), t(batch.k_start), t(batch.k_len)
    ql = np.full(batch.B, d.curr_len, np.int32)
    qs = np.concatenate([[0], np.cumsum(ql)[:-1]]).astype(np.int32)
    res = {}
    for D in (64, 128):
        K = inputs.randn((1, batch.total, 8, D), seed=1, device=dev)
        V = inputs.randn((1, batch.total, 8, D), seed=2, device=dev)
        Q = inputs.randn((1, batch.total, 32, D), seed=3, device=dev)
        O = torch.empty_like(Q)
        flops = 4.0 * D * 32 * _visible_pairs(role, seg, range(L), 0) * batch.B
        call = lambda ws=None: sonic.sonic_attn_prefill(
            Q, K, V, s_, r_, O, k_start=ks, k_len=kl, q_start=ks, q_len=kl, max_q_len=L,
            max_k_len=L, key_order=1, workspace=ws)
        ws = call()
        ms = _ev_time(lambda: call(ws))
        res[f"all_rows_retained_first_d{D}"] = {"ms": round(ms, 3),
                                                "tflops": round(flops / ms / 1e9, 1)}
        Qc = inputs.randn((1, int(ql.sum()), 32, D), seed=4, device=dev)
        Oc = torch.empty_like(Qc)
        flops = 4.0 * D * 32 * _visible_pairs(role, seg, range(L - d.curr_len, L), 0) * batch.B
        qst, qlt = t(qs), t(ql)
        call = lambda ws=None: sonic.sonic_attn_prefill(
            Qc, K, V, s_, r_, Oc, k_start=ks, k_len=kl, q_start=qst, q_len=qlt,
            max_q_len=int(ql.max()), max_k_len=L, key_order=1, workspace=ws)
        ws = call()
        ms = _ev_time(lambda: call(ws))
        res[f"current_rows_retained_first_d{D}"] = {"ms": round(ms, 3),
                                                    "tflops": round(flops / ms / 1e9, 1)}
    return {"workload": "masked prefill, batch 8 x 5632 rows, 32/8 heads, head_dim 64 and 128",
            "results": res}


def extra_decode():
    """Decode over retained caches: Llama-3-8B-like (batch 16, 32 layers, 32/8
    heads, 641 retained rows) and 64 long ragged dialogues with Nexus =
    len/2 and len/5 (32 layers, 32/8 heads)."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    t = lambda a: torch.as_tensor(np.asarray(a)).to(dev)
    res = {}
    lr2 = inputs.long_ragged(2)
    cases = {"llama8b_641_rows": inputs.decode_llama8b(),
             "long_ragged_nexus_len_div_2": lr2,
             "long_ragged_nexus_len_div_5": inputs.long_ragged(5),
             # head_dim 64 (CUDA-core kernel): the same dialogues, 8 layers, 32/8 heads
             "long_ragged_nexus_len_div_2_head_dim_64": (lr2[0], inputs.Heads(8, 32, 8, 64))}
    for name, (b2, h2) in cases.items():
        lens = np.array([x.recipe_retained + 1 for x in b2.dialogues], np.int32)
        starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int32)
        T = int(lens.sum())
        K = inputs.randn((h2.n_layers, T, h2.hkv, h2.d), seed=7, device=dev)
        V = inputs.randn((h2.n_layers, T, h2.hkv, h2.d), seed=8, device=dev)
        q = inputs.randn((h2.n_layers, b2.B, h2.hq, h2.d), seed=9, device=dev)
        O = torch.empty_like(q)
        lt, st = t(lens), t(starts)
        ms = _ev_time(lambda: sonic.sonic_attn_decode(q, K, V, lt, O, kv_start=st,
                                                      max_len=int(lens.max())), reps=10)
        by = (T * h2.hkv * h2.d * 2 * 2 + 2 * b2.B * h2.hq * h2.d * 2) * h2.n_layers
        res[name] = {"ms": round(ms, 3), "gbs": round(by / ms / 1e6, 1), "gb": round(by / 1e9, 2)}
        del K, V
        torch.cuda.empty_cache()
    return {"workload": "decode over retained caches", "results": res}


def extra_context(n_layers: int = 8):
    """Full-context vs SONIC decode at the mixed serving step's shapes: the 56
    decoding dialogues (28/4 heads, D = 128; n_layers of 28 layers) decode one
    token over (a) their whole dialogue without Nexus tokens -- system prompt,
    every turn, the current turn: plain causal attention -- and (b) their
    retained cache -- system prompt, Nexus tokens, current turn (Eq. 15).  The
    same kernel serves both; the ratio is the decode-side mechanism behind
    the paper's end-to-end speedup."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    t = lambda a: torch.as_tensor(np.asarray(a)).to(dev)
    ms_ = inputs.mixed_serving(seed=1)
    h = ms_.heads
    res = {}
    full = np.array([d.sys_len + sum(b for b, _ in d.segments) + d.curr_len + 1
                     for d in ms_.decode_hist], np.int64)
    ret = np.array([d.recipe_retained + 1 for d in ms_.decode_hist], np.int64)
    for name, lens in (("full_context", full), ("sonic_retained", ret)):
        lens = lens.astype(np.int32)
        starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int32)
        T = int(lens.sum())
        K = inputs.randn((n_layers, T, h.hkv, h.d), seed=7, device=dev)
        V = inputs.randn((n_layers, T, h.hkv, h.d), seed=8, device=dev)
        q = inputs.randn((n_layers, len(lens), h.hq, h.d), seed=9, device=dev)
        O = torch.empty_like(q)
        lt, st = t(lens), t(starts)
        ms = _ev_time(lambda: sonic.sonic_attn_decode(q, K, V, lt, O, kv_start=st,
                                                      max_len=int(lens.max())), reps=10)
        by = (T * h.hkv * h.d * 2 * 2 + 2 * len(lens) * h.hq * h.d * 2) * n_layers
        res[name] = {"rows": T, "ms": round(ms, 3), "gbs": round(by / ms / 1e6, 1),
                     "kv_gb": round(T * h.hkv * h.d * 4 * n_layers / 1e9, 2)}
        del K, V
        torch.cuda.empty_cache()
    res["speedup"] = round(res["full_context"]["ms"] / res["sonic_retained"]["ms"], 2)
    return {"workload": f"56 decoding dialogues of the mixed serving step, {n_layers} layers, "
                        "28/4 heads, D=128", "results": res}


def extra_nexus_gen(n_layers: int = 0):
    """Nexus generation with incremental compaction (Sec. 3.1, Table 3's
    "Nexus Gen." step) at the masked-prefill shapes: batch 8, 32 layers, 32/8
    heads, D = 128, 512 system tokens, 16 segments of 256 body + 32 Nexus.
    Segment i: the 32 Nexus rows attend over [retained | body_i | Nexus_i]
    (one prefill launch for the batch and all layers), then compaction drops
    body_i.  Inputs of every segment step are staged beforehand; the timed
    region is the 16 prefill and 16 compaction launches.  n_layers > 0 runs
    that many layers instead of 32 (small profiler captures)."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    t = lambda a: torch.as_tensor(np.asarray(a)).to(dev)
    batch, hd = inputs.masked_prefill()
    d = batch.dialogues[0]
    B, NL = batch.B, (n_layers if n_layers > 0 else hd.n_layers)
    sysl, segs = d.sys_len, d.segments
    steps = []
    flops = comp_bytes = pf_bytes = 0.0
    for i, (nb, nk) in enumerate(segs, start=1):
        r_len = sysl + sum(k for _, k in segs[:i - 1])
        L = r_len + nb + nk
        role = np.concatenate([np.zeros(sysl, np.uint8), np.full(r_len - sysl, 2, np.uint8),
                               np.full(nb, 1, np.uint8), np.full(nk, 2, np.uint8)])
        seg = np.concatenate([np.zeros(sysl, np.int32),
                              np.repeat(np.arange(1, i, dtype=np.int32), [k for _, k in segs[:i - 1]]),
                              np.full(nb + nk, i, np.int32)])
        K = inputs.randn((NL, B * L, hd.hkv, hd.d), seed=100 + i, device=dev)
        V = inputs.randn((NL, B * L, hd.hkv, hd.d), seed=200 + i, device=dev)
        Q = inputs.randn((NL, B * nk, hd.hq, hd.d), seed=300 + i, device=dev)
        O = torch.empty_like(Q)
        ks = t(np.arange(B, dtype=np.int32) * L)
        kl = t(np.full(B, L, np.int32))
        qs = t(np.arange(B, dtype=np.int32) * nk)
        ql = t(np.full(B, nk, np.int32))
        R = r_len + nk
        oK = torch.empty((NL, B * R, hd.hkv, hd.d), dtype=K.dtype, device=dev)
        oV = torch.empty_like(oK)
        off = torch.zeros(B + 1, dtype=torch.int32, device=dev)
        steps.append(dict(K=K, V=V, Q=Q, O=O, ks=ks, kl=kl, qs=qs, ql=ql, L=L, nk=nk,
                          role=t(np.tile(role, B)), seg=t(np.tile(seg, B)), oK=oK, oV=oV, off=off))
        flops += 4.0 * hd.d * hd.hq * _visible_pairs(role, seg, range(L - nk, L), 0) * B * NL
        comp_bytes += 2.0 * R * B * hd.hkv * hd.d * 2 * 2 * NL
        # the prefill's bytes: every key row is visible to the Nexus rows, so K and
        # V of all L rows are read once per KV head, Q read and O written once
        pf_bytes += (2.0 * L * hd.hkv + 2.0 * nk * hd.hq) * B * hd.d * 2 * NL

    def prefills():
        for s in steps:
            s["ws_p"] = sonic.sonic_attn_prefill(
                s["Q"], s["K"], s["V"], s["seg"], s["role"], s["O"], k_start=s["ks"],
                k_len=s["kl"], q_start=s["qs"], q_len=s["ql"], max_q_len=s["nk"],
                max_k_len=s["L"], workspace=s.get("ws_p"))

    def compactions():
        for s in steps:
            s["ws_c"] = sonic.sonic_compact_kv(s["K"], s["V"], s["seg"], s["role"], s["oK"],
                                               s["oV"], s["off"], k_start=s["ks"], k_len=s["kl"],
                                               workspace=s.get("ws_c"))

    p_ms = _ev_time(prefills)
    c_ms = _ev_time(compactions)
    pk = _peaks()
    # 32 query rows of 4 heads per K/V row: the prefill is bound by HBM, not by
    # the tensor cores (flops per byte below the ridge point peak_bf16 / peak_hbm)
    intensity = flops / pf_bytes
    return {"workload": f"Nexus generation: batch 8, {NL} layers, 32/8 heads, D=128, "
                        "16 segments of 256 body + 32 Nexus after 512 system tokens",
            "results": {"prefill_ms_all_segments": round(p_ms, 3),
                        "prefill_tflops": round(flops / p_ms / 1e9, 1),
                        "prefill_frac_of_bf16_peak": round(flops / p_ms / 1e9 / pk["bf16"], 4),
                        "prefill_gb": round(pf_bytes / 1e9, 3),
                        "prefill_gbs": round(pf_bytes / p_ms / 1e6, 1),
                        "prefill_flops_per_byte": round(intensity, 1),
                        "prefill_roofline": {
                            "bound": "hbm", "peak": pk["hbm"], "unit": "GB/s",
                            "frac": round(pf_bytes / p_ms / 1e6 / pk["hbm"], 4),
                            "tflops_at_peak_hbm": round(intensity * pk["hbm"] / 1e3, 1)},
                        "compaction_ms_all_segments": round(c_ms, 3),
                        "compaction_gbs": round(comp_bytes / c_ms / 1e6, 1),
                        "ms_per_segment": round((p_ms + c_ms) / len(segs), 3)}}


def extra_decode_graph():
    """Decode of the Llama-3-8B-like batch (16 x 641 retained rows, 32 layers,
    32/8 heads): one launch over all layers, and 32 per-layer launches
    captured once in a CUDA graph and replayed."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    b2, h2 = inputs.decode_llama8b()
    lens = np.array([x.recipe_retained + 1 for x in b2.dialogues], np.int32)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int32)
    T, nl = int(lens.sum()), h2.n_layers
    K = inputs.randn((nl, T, h2.hkv, h2.d), seed=7, device=dev)
    V = inputs.randn((nl, T, h2.hkv, h2.d), seed=8, device=dev)
    q = inputs.randn((nl, b2.B, h2.hq, h2.d), seed=9, device=dev)
    O = torch.empty_like(q)
    lt = torch.as_tensor(lens).to(dev)
    st = torch.as_tensor(starts).to(dev)
    ml = int(lens.max())
    ws_all = sonic.sonic_attn_decode(q, K, V, lt, O, kv_start=st, max_len=ml)
    ms_all = _ev_time(lambda: sonic.sonic_attn_decode(q, K, V, lt, O, kv_start=st, max_len=ml,
                                                      workspace=ws_all), reps=20, warm=3)
    ws = [sonic.sonic_attn_decode(q[l:l + 1], K[l:l + 1], V[l:l + 1], lt, O[l:l + 1],
                                  kv_start=st, max_len=ml) for l in range(nl)]
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for l in range(nl):
            sonic.sonic_attn_decode(q[l:l + 1], K[l:l + 1], V[l:l + 1], lt, O[l:l + 1],
                                    kv_start=st, max_len=ml, workspace=ws[l])
    ms_graph = _ev_time(g.replay, reps=20, warm=3)
    ms_eager = _ev_time(lambda: [sonic.sonic_attn_decode(
        q[l:l + 1], K[l:l + 1], V[l:l + 1], lt, O[l:l + 1], kv_start=st, max_len=ml,
        workspace=ws[l]) for l in range(nl)], reps=20, warm=3)
    by = (T * h2.hkv * h2.d * 2 * 2 + 2 * b2.B * h2.hq * h2.d * 2) * nl
    rate = lambda ms: round(by / ms / 1e6, 1)
    return {"workload": "decode, batch 16 x 641 retained rows, 32 layers, 32/8 heads, D=128 "
                        "(1.35 GB)",
            "results": {"one_launch_all_layers": {"ms": round(ms_all, 4), "gbs": rate(ms_all)},
                        "per_layer_launches_cuda_graph": {"ms": round(ms_graph, 4),
                                                          "gbs": rate(ms_graph)},
                        "per_layer_launches_eager": {"ms": round(ms_eager, 4),
                                                     "gbs": rate(ms_eager)}}}


def extra_compaction():
    """KV compaction (Sec. 3.2 body removal) at the masked-prefill shapes
    (batch 8 x 5632 raw rows -> 1536 retained, 32 layers, 8 KV heads, D = 128:
    3.22 GB moved) and of the long ragged histories (64 dialogues, Nexus =
    len/2 and len/5, 4 of the 32 layers: the per-layer work is the same)."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    t = lambda a: torch.as_tensor(np.asarray(a)).to(dev)
    res = {}
    cases = [("masked_prefill_32_layers", inputs.masked_prefill(), 32),
             ("long_ragged_nexus_len_div_2_4_layers", inputs.long_ragged(2), 4),
             ("long_ragged_nexus_len_div_5_4_layers", inputs.long_ragged(5), 4)]
    for name, (batch, hd), nl in cases:
        K = inputs.randn((nl, batch.total, hd.hkv, hd.d), seed=5, device=dev)
        V = inputs.randn((nl, batch.total, hd.hkv, hd.d), seed=6, device=dev)
        ret = sum(d.recipe_retained for d in batch.dialogues)
        oK = torch.empty((nl, ret, hd.hkv, hd.d), dtype=K.dtype, device=dev)
        oV = torch.empty_like(oK)
        off = torch.zeros(batch.B + 1, dtype=torch.int32, device=dev)
        r_, s_, ks, kl = t(batch.role), t(batch.seg), t(batch.k_start), t(batch.k_len)
        ws = sonic.sonic_compact_kv(K, V, s_, r_, oK, oV, off, k_start=ks, k_len=kl)
        ms = _ev_time(lambda: sonic.sonic_compact_kv(K, V, s_, r_, oK, oV, off, k_start=ks,
                                                     k_len=kl, workspace=ws), reps=10, warm=3)
        by = 2.0 * ret * hd.hkv * hd.d * 2 * 2 * nl
        res[name] = {"ms": round(ms, 3), "gbs": round(by / ms / 1e6, 1), "gb_moved": round(by / 1e9, 2),
                     "raw_gb": round(2.0 * batch.total * hd.hkv * hd.d * 2 * nl / 1e9, 2)}
        del K, V, oK, oV
        torch.cuda.empty_cache()
    return {"workload": "KV compaction (retained rows read + written, K and V)", "results": res}


def extra_nexus_mass():
    """Cost of the attention-mass output (Sec. 4.1 Eq. 9's A_nexus per row and
    head) on the mixed serving step at 8 layers: its prefill and its decode
    launch, each with and without the mass (same inputs, same outputs
    otherwise)."""
    import torch
    dev = torch.device("cuda", 0)
    lay = Layout(n_layers=8)
    g = GpuStep(lay, dev)
    sonic = g.sonic
    mass_p = torch.empty((lay.NL, lay.T_q, lay.HQ), dtype=torch.float32, device=dev)
    mass_d = torch.empty((lay.NL, lay.n_dec, lay.HQ), dtype=torch.float32, device=dev)

    def prefill(m):
        sonic.sonic_attn_prefill(
            g.Qp, g.Kret, g.Vret, g.seg_ret, g.role_ret, g.Op, k_start=g.k_start_pre,
            k_len=g.k_len_pre, q_start=g.q_start, q_len=g.q_len,
            max_q_len=int(lay.q_len.max()), max_k_len=int(lay.k_len_pre.max()), nexus_mass=m)

    def decode(m):
        sonic.sonic_attn_decode(g.qd, g.Kret, g.Vret, g.dec_len, g.Od, kv_start=g.dec_start,
                                max_len=int(lay.dec_len.max()), role=g.role_ret, nexus_mass=m)

    res = {}
    for name, fn, m in (("prefill", prefill, mass_p), ("decode", decode, mass_d)):
        t0 = _ev_time(lambda: fn(None), reps=10)
        t1 = _ev_time(lambda: fn(m), reps=10)
        res[name] = {"ms": round(t0, 3), "ms_with_mass": round(t1, 3),
                     "overhead_pct": round(100.0 * (t1 / t0 - 1.0), 1)}
    pf = lay.prefill_flops()
    res["prefill"]["tflops_with_mass"] = round(pf / res["prefill"]["ms_with_mass"] / 1e9, 1)
    res["decode"]["gbs_with_mass"] = round(lay.decode_bytes() / res["decode"]["ms_with_mass"] / 1e6, 1)
    return {"workload": "mixed serving step, 8 layers: prefill and decode with / without the "
                        "attention mass on Nexus keys", "results": res}


def extra_routed():
    """Role-routed projections (Sec. 3.1): the QKV projection of a Nexus
    generation segment step (8 x (256 body + 32 Nexus) rows, Llama-3-8B-like
    4096 -> 4096 + 1024 + 1024, K/V into cache rows), the QKV and O
    projections of the serving step's 12,146 prefill rows (Qwen2.5-7B-like
    3584 -> 3584 + 512 + 512, and 3584 -> 3584), with half of those rows
    marked Nexus in runs of 32, and the QKV projection of the same rows as
    one current turn (one role: no rows are copied).  Beside each: cuBLAS
    (torch.matmul) on the role groups plus the row scatter, as context."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    bf = torch.bfloat16
    res = {}
    nexus_gen = np.tile(np.r_[np.full(256, 1), np.full(32, 2)], 8).astype(np.uint8)
    serving = np.repeat(np.tile(np.array([3, 2], np.uint8), 12146 // 64 + 1), 32)[:12146]
    cases = {
        "nexus_gen_qkv_T2304_4096x6144": (nexus_gen, 4096, [4096, 1024, 1024], [0, 1, 1]),
        "serving_qkv_T12146_3584x4608": (serving, 3584, [3584, 512, 512], [0, 1, 1]),
        "serving_o_T12146_3584x3584": (serving, 3584, [3584], [0]),
        "current_turn_qkv_T12146_3584x4608": (np.full(12146, 3, np.uint8), 3584,
                                              [3584, 512, 512], [0, 1, 1]),
    }
    for name, (role, d_in, cols, scat) in cases.items():
        T, d_out = len(role), sum(cols)
        X = inputs.randn((T, d_in), seed=1, device=dev)
        W = inputs.randn((d_out, d_in), seed=2, device=dev)
        Wn = inputs.randn((d_out, d_in), seed=3, device=dev)
        role_t = torch.as_tensor(role).to(dev)
        cache_rows = 2 * T
        dst = torch.as_tensor(np.random.default_rng(0).permutation(cache_rows)[:T].astype(
            np.int32)).to(dev)
        outs = [torch.empty((cache_rows if s else T, c), dtype=bf, device=dev)
                for c, s in zip(cols, scat)]
        parts = list(zip(outs, [bool(s) for s in scat]))
        ws = sonic.sonic_routed_linear(X, W, Wn, role_t, parts, dst_row=dst)
        ms = _ev_time(lambda: sonic.sonic_routed_linear(X, W, Wn, role_t, parts, dst_row=dst,
                                                        workspace=ws), reps=10, warm=3)
        nex = torch.as_tensor(np.nonzero(role == 2)[0]).to(dev)
        oth = torch.as_tensor(np.nonzero(role != 2)[0]).to(dev)
        dstl = dst.long()

        def cublas():
            y = torch.empty((T, d_out), dtype=bf, device=dev)
            y[oth] = X[oth] @ W.T
            y[nex] = X[nex] @ Wn.T
            c0 = 0
            for out, s in zip(outs, scat):
                if s:
                    out[dstl] = y[:, c0:c0 + out.shape[1]]
                else:
                    out.copy_(y[:, c0:c0 + out.shape[1]])
                c0 += out.shape[1]
        ms_ref = _ev_time(cublas, reps=10, warm=3)
        ms_mm = _ev_time(lambda: torch.matmul(X, W.T), reps=10, warm=3)
        fl = 2.0 * T * d_in * d_out
        res[name] = {"ms": round(ms, 4), "tflops": round(fl / ms / 1e9, 1),
                     "cublas_grouped_scatter_ms": round(ms_ref, 4),
                     "cublas_one_matmul_ms": round(ms_mm, 4),
                     "cublas_one_matmul_tflops": round(fl / ms_mm / 1e9, 1)}
        del X, W, Wn, outs, ws
        torch.cuda.empty_cache()
    return {"workload": "role-routed QKV / O projections (bf16, fp32 accumulate)", "results": res}


# ---------------------------------------------------------------------------
# The named workloads other than the serving step, timed after it in the
# default run (`configs` object of the JSON line)
# ---------------------------------------------------------------------------

def _free_cuda():
    import gc
    import torch
    gc.collect()
    torch.cuda.empty_cache()


def _decode_rate(b2, h2, n_layers: int, reps: int = 10):
    """One decode step over the retained caches of dialogues `b2` (recipe
    lengths + the new token) for n_layers layers in one launch.  Returns
    (ms per launch, algorithmic bytes, GB/s)."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    lens = np.array([x.recipe_retained + 1 for x in b2.dialogues], np.int32)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int32)
    T = int(lens.sum())
    K = inputs.randn((n_layers, T, h2.hkv, h2.d), seed=7, device=dev)
    V = inputs.randn((n_layers, T, h2.hkv, h2.d), seed=8, device=dev)
    q = inputs.randn((n_layers, b2.B, h2.hq, h2.d), seed=9, device=dev)
    O = torch.empty_like(q)
    lt = torch.as_tensor(lens).to(dev)
    st = torch.as_tensor(starts).to(dev)
    ws = sonic.sonic_attn_decode(q, K, V, lt, O, kv_start=st, max_len=int(lens.max()))
    ms = _ev_time(lambda: sonic.sonic_attn_decode(q, K, V, lt, O, kv_start=st,
                                                  max_len=int(lens.max()), workspace=ws),
                  reps=reps, warm=3)
    by = float(T * h2.hkv * h2.d * 2 * 2 + 2 * b2.B * h2.hq * h2.d * 2 + b2.B * 8) * n_layers
    del K, V, q, O, ws
    _free_cuda()
    return ms, by, by / ms / 1e6


def config_workloads():
    """The decode, masked-prefill and long-ragged workloads at full size on
    one GPU, each against its roofline (measured peaks): decode and
    compaction in HBM GB/s, prefill in algorithmic TFLOP/s (visible pairs
    only; the kernel is timed alone, so against the burst bf16 peak).  Every
    input is larger than L2 except where noted."""
    import torch
    from paper_2601_21927_gb300 import inputs, sonic
    dev = torch.device("cuda", 0)
    pk = _peaks()
    t = lambda a: torch.as_tensor(np.asarray(a)).to(dev)
    hbm = lambda gbs: {"bound": "hbm", "peak": pk["hbm"], "unit": "GB/s",
                       "frac": round(gbs / pk["hbm"], 4)}
    out = {}

    # decode, Llama-3-8B-like: 16 x 641 retained rows, 32 layers, 32/8 heads
    b2, h2 = inputs.decode_llama8b()
    ms, by, gbs = _decode_rate(b2, h2, h2.n_layers)
    out["decode_llama8b"] = {
        "workload": "decode, batch 16 x 641 retained rows (256 system, 8 x 32 Nexus, 128 current, "
                    "1 new), 32 layers in one launch, 32/8 heads, D=128, bf16",
        "ms": round(ms, 4), "gb": round(by / 1e9, 3), "value": round(gbs, 1), "unit": "GB/s",
        "roofline": hbm(gbs)}

    # masked prefill: 8 x 5632 rows, every row a query, full mask, all 32 layers
    # in one launch (and one layer alone); then the current turn's rows alone;
    # then compaction of all 32 layers
    batch, hd = inputs.masked_prefill()
    d = batch.dialogues[0]
    role, seg = d.arrays()
    L = d.length
    NL = hd.n_layers
    K = inputs.randn((NL, batch.total, hd.hkv, hd.d), seed=1, device=dev)
    V = inputs.randn((NL, batch.total, hd.hkv, hd.d), seed=2, device=dev)
    Q = inputs.randn((NL, batch.total, hd.hq, hd.d), seed=3, device=dev)
    O = torch.empty_like(Q)
    r_, s_, ks, kl = t(batch.role), t(batch.seg), t(batch.k_start), t(batch.k_len)
    flops1 = 4.0 * hd.d * hd.hq * _visible_pairs(role, seg, range(L), 0) * batch.B
    res = {}

    def timed(name, Qx, Ox, nl, fl, order, q_start, q_len, max_q):
        call = lambda ws=None: sonic.sonic_attn_prefill(
            Qx[:nl], K[:nl], V[:nl], s_, r_, Ox[:nl], k_start=ks, k_len=kl, q_start=q_start,
            q_len=q_len, max_q_len=max_q, max_k_len=L, key_order=order, workspace=ws)
        ws = call()
        sampler = ClockSampler(0)
        sampler.start()
        ms = _ev_time(lambda: call(ws), reps=10, warm=3)
        clk = sampler.stop()
        tf = fl * nl / ms / 1e9
        res[name] = {"layers": nl, "ms": round(ms, 4), "value": round(tf, 1), "unit": "TFLOP/s",
                     "frac": round(tf / pk["bf16"], 4),
                     "frac_of_sustained": round(tf / pk["bf16_sus"], 4), "clocks": clk}
        del ws

    for order, oname in ((1, "retained_first"), (0, "as_given")):
        timed(f"all_rows_{oname}", Q, O, NL, flops1, order, ks, kl, L)
    timed("all_rows_retained_first_one_layer", Q, O, 1, flops1, 1, ks, kl, L)
    ql = np.full(batch.B, d.curr_len, np.int32)
    qs = np.concatenate([[0], np.cumsum(ql)[:-1]]).astype(np.int32)
    Qc = Q[:, :int(ql.sum())]
    Oc = torch.empty_like(Qc)
    cflops = 4.0 * hd.d * hd.hq * _visible_pairs(role, seg, range(L - d.curr_len, L), 0) * batch.B
    qst, qlt = t(qs), t(ql)
    for order, oname in ((1, "retained_first"), (0, "as_given")):
        timed(f"current_rows_{oname}", Qc, Oc, NL, cflops, order, qst, qlt, int(ql.max()))
    del K, V, Q, O, Qc, Oc
    _free_cuda()
    head = res["all_rows_retained_first"]
    prefill = {"workload": "masked prefill, batch 8 x 5632 rows (512 system, 16 x (256 body + 32 "
                           "Nexus), 512 current), every row a query, full Sec. 3.2 mask, 32/8 "
                           "heads, D=128, bf16, 32 layers in one launch; retained-first order "
                           "(its key and query order and K/V copies included)",
               "flops": flops1 * NL, "ms": head["ms"], "value": head["value"], "unit": "TFLOP/s",
               "roofline": {"bound": "tensor", "peak": pk["bf16"], "unit": "TFLOP/s",
                            "frac": head["frac"], "peak_source": pk["source"] + " bf16 burst",
                            "peak_sustained": pk["bf16_sus"],
                            "frac_of_sustained": head["frac_of_sustained"]},
               "clocks": head["clocks"], "variants": res}
    # compaction of all 32 layers' K/V (raw 5.91 GB in, 3.22 GB moved)
    K = inputs.randn((hd.n_layers, batch.total, hd.hkv, hd.d), seed=5, device=dev)
    V = inputs.randn((hd.n_layers, batch.total, hd.hkv, hd.d), seed=6, device=dev)
    ret = sum(x.recipe_retained for x in batch.dialogues)
    oK = torch.empty((hd.n_layers, ret, hd.hkv, hd.d), dtype=K.dtype, device=dev)
    oV = torch.empty_like(oK)
    off = torch.zeros(batch.B + 1, dtype=torch.int32, device=dev)
    ws = sonic.sonic_compact_kv(K, V, s_, r_, oK, oV, off, k_start=ks, k_len=kl)
    ms = _ev_time(lambda: sonic.sonic_compact_kv(K, V, s_, r_, oK, oV, off, k_start=ks,
                                                 k_len=kl, workspace=ws), reps=10, warm=3)
    by = 2.0 * ret * hd.hkv * hd.d * 2 * 2 * hd.n_layers
    prefill["compaction"] = {"ms": round(ms, 4), "gb": round(by / 1e9, 3),
                             "value": round(by / ms / 1e6, 1), "unit": "GB/s",
                             "roofline": hbm(by / ms / 1e6)}
    del K, V, oK, oV, ws
    _free_cuda()
    out["masked_prefill"] = prefill

    # long ragged dialogues: 64 sequences, 32 layers, both Nexus budgets
    for div in (2, 5):
        b4, h4 = inputs.long_ragged(div)
        ms, by, gbs = _decode_rate(b4, h4, h4.n_layers)
        out[f"long_ragged_decode_nexus_len_div_{div}"] = {
            "workload": f"decode, 64 ragged dialogues (turns U[4,32] of U[64,1024] tokens, Nexus "
                        f"= ceil(len/{div}), 256 system), 32 layers in one launch, 32/8 heads, "
                        f"D=128, bf16",
            "ms": round(ms, 4), "gb": round(by / 1e9, 3), "value": round(gbs, 1), "unit": "GB/s",
            "roofline": hbm(gbs)}
    return out


EXTRAS = {"masked_prefill": extra_masked_prefill, "decode": extra_decode,
          "nexus_mass": extra_nexus_mass, "routed": extra_routed, "compaction": extra_compaction,
          "decode_graph": extra_decode_graph, "prefill_d64": extra_prefill_d64,
          "context": extra_context, "nexus_gen": extra_nexus_gen}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="sonic", choices=["sonic", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other named workloads after the serving step")
    ap.add_argument("--only", choices=["compact", "prefill", "decode"], default=None,
                    help="time one phase alone (for profiler captures)")
    ap.add_argument("--layers", type=int, default=0, help="override the layer count")
    ap.add_argument("--extra", choices=sorted(EXTRAS), default=None,
                    help="time a further workload instead of the benchmark step")
    args = ap.parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))

    if args.extra:
        if rank == 0:
            kw = {"n_layers": args.layers} if args.layers and args.extra == "nexus_gen" else {}
            out = EXTRAS[args.extra](**kw)
            out["extra"] = args.extra
            print(json.dumps(out))
        return

    if args.impl == "reference":
        if rank != 0:
            return
        lay = Layout()
        per_step, vals = [], []
        for i in range(args.warmup + args.steps):
            v, dt, cores, desc = oracle_sample(lay)
            if i >= args.warmup:
                per_step.append(dt)
                vals.append(v)
        value = float(np.mean(vals))
        out = {"metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
               "steps": args.steps, "warmup": args.warmup,
               "ms_per_step": round(1e3 * float(np.mean(per_step)), 1),
               "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
               "dtype": "f64", "data": "synthetic", "impl": "reference",
               "config": {"workload": WORKLOAD, "sample": desc},
               "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cores,
                                "kind": "oracle", "sample": desc},
               "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                       "d2h_bytes_per_step": 0}}
        print(json.dumps(out))
        return

    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    out, lay = run_gpu(args, rank, world)
    if rank == 0 and world == 1 and not args.only and not args.no_configs:
        _free_cuda()
        out["configs"] = config_workloads()
    if rank == 0 and world == 1 and not args.no_cpu_baseline and not args.only:
        v, dt, cores, desc = oracle_sample(lay)
        dv, ddt, dcores, ddesc = oracle_decode_sample(lay)
        cv, cdt, ccores, cdesc = oracle_compact_sample(lay)
        out["cpu_baseline"] = {
            "value": v, "unit": "TFLOP/s", "cores": cores, "kind": "oracle", "sample": desc,
            "seconds": round(dt, 2),
            "decode": {"value": round(dv, 4), "unit": "GB/s", "cores": dcores, "kind": "oracle",
                       "sample": ddesc, "seconds": round(ddt, 2)},
            "compaction": {"value": round(cv, 4), "unit": "GB/s", "cores": ccores,
                           "kind": "oracle", "sample": cdesc, "seconds": round(cdt, 2)}}
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(out))


if __name__ == "__main__":
    main()
