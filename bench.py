"""Benchmark of the keyed-race hot path on GB300.

One step = pps_draft_list over every draft row + pps_verify_tree over every
node row (target race, tree walk, watermark scores) of one batch of
synthetic logits.  Default workload: B=64 sequences, V=128256, K=8 drafts,
gamma=5 (K chains of depth 5 = 41 nodes per sequence: 2,624 target rows and
2,112 draft rows), bf16 Zipf(1.0) logits under a random vocabulary
permutation per row, draft = target + N(0,1).  Inputs (1.21 GB) exceed L2
(129 MB), so no flush is needed between steps.

`value` counts row-passes per second (draft rows + target rows, all ranks).
`--impl reference` times the CPU oracle on a bounded sample of the same rows.
The default line's `parity` key compares every row of the step with the oracle
(run in the cpu_baseline leg, after the device-timed region).
"""
from __future__ import annotations

import argparse
import json
import os
import platform
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verified rows/s and GB/s vs HBM peak at V=128256, K=8, B=64 (1xGB300)"
WIDE_MULS_PER_SM_CLK = 32
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "race_kernel_zipf_k8_traffic.txt")
TRUNC_TRAFFIC_FILE = os.path.join(ROOT, "profiles", "trunc_kernel_zipf_k8_top50_traffic.txt")


def kernel_source_digest() -> str:
    """sha1 over the CUDA sources of libpps (a recorded ncu figure is stale once this changes)."""
    import hashlib
    h = hashlib.sha1()
    csrc = os.path.join(ROOT, "paper_2609_21858_gb300", "csrc")
    for name in ("pps_race.cu", "pps_device.cuh", "pps_internal.h", "pps_trunc.cuh"):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()


def philox_only_rate(dev) -> float:
    """Tokens per second of the keyed source alone (4 tokens per Philox block)."""
    from paper_2609_21858_gb300 import pps
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    out_len = sms * 8 * 256
    n_blocks = out_len * 512
    for _ in range(3):
        pps.selftest_philox_rate(n_blocks, out_len)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(5):
        pps.selftest_philox_rate(n_blocks, out_len)
    e1.record()
    torch.cuda.synchronize(dev)
    return 5 * 4 * n_blocks / (e0.elapsed_time(e1) / 1e3)


def _traffic(which: str, path: str = TRAFFIC_FILE):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current kernel."""
    try:
        kv = {}
        with open(path) as f:
            for line in f:
                if "=" in line and not line.startswith("#"):
                    k, v = line.strip().split("=", 1)
                    kv[k.strip()] = v.strip()
        if kv.get("kernel_source_sha1") != kernel_source_digest():
            return None
        return float(kv[f"{which}_dram_bytes_per_launch"])
    except Exception:
        return None


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class Clocks:
    """nvidia-smi sampling during the timed region."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                p = [x.strip() for x in line.split(",")]
                if len(p) < 9:
                    continue
                try:
                    sm.append(float(p[1]))
                    smax.append(float(p[2]))
                except ValueError:
                    continue
                for n, v in zip(names, p[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_init():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(local)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def cpu_model() -> str:
    """The host CPU's name (x86 'model name', else the Arm implementer/part), for the oracle timing."""
    try:
        info = open("/proc/cpuinfo").read()
        for line in info.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
        parts = {}
        for line in info.splitlines():
            if ":" in line:
                k, v = line.split(":", 1)
                parts.setdefault(k.strip(), v.strip())
        if "CPU part" in parts:
            return f"{platform.machine()} implementer {parts.get('CPU implementer')} part {parts['CPU part']}"
    except OSError:
        pass
    return platform.machine()


def race_workload_name(args, wl) -> str:
    """The config's workload string of a race workload (both arms print the same one)."""
    t = wl.tree
    trunc = f", top-k {args.top_k}, top-p {args.top_p}" if args.top_k > 0 else ""
    return (f"{args.workload}: B={t.n_seq}, V={wl.vocab}, K={t.K}, gamma={t.gamma}, "
            f"{t.n_nodes} target rows + {t.n_draft} draft rows per step{trunc}")


def oracle_sample(wl, n_draft_rows: int, n_target_rows: int, seed: int = 0, top_k: int = 0, top_p: float = 1.0,
                  keep: dict | None = None):
    """Host copies of a bounded sample of the workload's rows and a timer over them.  A sample as
    large as the step takes every row in order; `keep` (a dict) then receives the oracle's lists
    and winners of the last run."""
    import oracle
    from paper_2609_21858_gb300 import synth
    t = wl.tree
    rng = np.random.default_rng(seed)
    if n_draft_rows >= t.n_draft and n_target_rows >= t.n_nodes:
        dr, nr = np.arange(t.n_draft), np.arange(t.n_nodes)
    else:
        dr = np.sort(rng.choice(t.n_draft, min(n_draft_rows, t.n_draft), replace=False))
        nr = np.sort(rng.choice(t.n_nodes, min(n_target_rows, t.n_nodes), replace=False))
    dsel = torch.as_tensor(dr, device=wl.q_logits.device)
    nsel = torch.as_tensor(nr, device=wl.p_logits.device)
    q = wl.q_logits[dsel].float().cpu().numpy()
    p = wl.p_logits[nsel].float().cpu().numpy()
    ids_d = (synth.u64(wl.draft_key[dsel]), synth.u64(wl.draft_ctx[dsel]), synth.u32(wl.draft_pos[dsel]))
    ids_n = (synth.u64(wl.node_key[nsel]), synth.u64(wl.node_ctx[nsel]), synth.u32(wl.node_pos[nsel]))
    rk = t.row_k[dr]
    cores = oracle.set_threads(0)

    def run():
        t0 = time.perf_counter()
        qq, pp = q, p
        if top_k > 0:
            qq, _ = oracle.truncate_rows(q, top_k, top_p)
            pp, _ = oracle.truncate_rows(p, top_k, top_p)
        d = oracle.draft_rows(qq, *ids_d, t.K, row_k=rk)
        w = oracle.target_rows(pp, *ids_n)
        dt = time.perf_counter() - t0
        if keep is not None:
            keep.update(draft=d, target=w)
        return dt

    return run, len(dr), len(nr), cores


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="zipf_k8")
    ap.add_argument("--k", type=int, default=8, help="drafts per root of the ksweep workload (1..32)")
    ap.add_argument("--n-seq", type=int, default=None, help="override the number of sequences (smaller profiling cases)")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--n-tokens", type=int, default=10_000_000, help="detector workload size")
    ap.add_argument("--top-k", type=int, default=0, help="truncate every row to its top-k set before the race")
    ap.add_argument("--top-p", type=float, default=1.0, help="then to its top-p set (with --top-k)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--philox-rounds", type=int, default=10, choices=[7, 10],
                    help="keyed source of the run: Philox4x32-10 (libpps.so) or -7 (libpps_r7.so)")
    ap.add_argument("--no-philox7", action="store_true",
                    help="default workload: skip the second measurement with the Philox4x32-7 build")
    ap.add_argument("--eager", action="store_true",
                    help="tree workloads: launch every call from Python instead of replaying a CUDA graph")
    args = ap.parse_args()

    rank, world, local = dist_init()
    from paper_2609_21858_gb300 import synth

    if args.impl == "reference":
        if rank != 0:
            return
        if args.philox_rounds != 10:
            import oracle
            oracle.set_philox_rounds(args.philox_rounds)
        run_reference(args, world)
        return

    from paper_2609_21858_gb300 import pps
    pps.use_library(args.philox_rounds)
    pps.lib()
    if args.philox_rounds != 10 and not args.no_cpu_baseline:
        import oracle
        oracle.set_philox_rounds(args.philox_rounds)
    dev = torch.device("cuda", local)
    if args.workload == "detector":
        run_detector(args, rank, world, dev)
        return
    if args.workload == "dynamic":
        run_dynamic(args, rank, world, dev)
        return
    if args.workload == "hetero":
        run_hetero(args, rank, world, dev)
        return
    if args.workload == "lmhead":
        run_lmhead(args, rank, world, dev)
        return
    wl = synth.make_workload(args.workload, device=dev, n_seq=args.n_seq,
                             K_sweep=args.k if args.workload == "ksweep" else None)
    t = wl.tree
    g = lambda x: torch.as_tensor(np.asarray(x)).to(dev).contiguous()
    row_k, seq_off, ndr, child = g(t.row_k), g(t.seq_off), g(t.node_draft_row), g(t.child_node)
    dk, dc, dp = wl.draft_key, wl.draft_ctx, wl.draft_pos
    nk, nc, np_ = wl.node_key, wl.node_ctx, wl.node_pos
    ws_d = pps.workspace(t.n_draft, 0, dev)
    ws_v = pps.workspace(t.n_nodes, t.n_seq, dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    dout = dict(tok=torch.empty(t.n_draft, t.K, dtype=torch.int32, device=dev), key=None,
                mult=torch.empty(t.n_draft, t.K, dtype=torch.int32, device=dev),
                ndist=torch.empty(t.n_draft, dtype=torch.int32, device=dev), samples=None)
    W = t.gamma + 1
    vout = dict(winner=torch.empty(t.n_nodes, dtype=torch.int32, device=dev),
                word=torch.empty(t.n_nodes, dtype=torch.int32, device=dev),
                accept_len=torch.empty(t.n_seq, dtype=torch.int32, device=dev),
                n_emitted=torch.empty(t.n_seq, dtype=torch.int32, device=dev),
                emitted=torch.empty(t.n_seq, W, dtype=torch.int32, device=dev),
                score=torch.empty(t.n_seq, W, dtype=torch.float32, device=dev),
                score_sum=torch.empty(t.n_seq, dtype=torch.float64, device=dev))
    stream = torch.cuda.current_stream(dev)

    def draft(q):
        pps.draft_list(q, dk, dc, dp, t.K, row_k=row_k, ws=ws_d, status=status, out=dout, stream=stream,
                       top_k=args.top_k, top_p=args.top_p)

    def verify(p):
        pps.verify_tree(p, nk, nc, np_, t.gamma, seq_off, ndr, dout["tok"], dout["ndist"], child, ws=ws_v,
                        status=status, out=vout, stream=stream, top_k=args.top_k, top_p=args.top_p)

    def step(q, p, ev=None):
        if ev is not None:
            ev[0].record(stream)
        draft(q)
        if ev is not None:
            ev[1].record(stream)
        verify(p)
        if ev is not None:
            ev[2].record(stream)

    q, p = wl.q_logits, wl.p_logits
    in_bytes = q.numel() * q.element_size() + p.numel() * p.element_size()
    l2 = getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 129 * 2 ** 20) or 129 * 2 ** 20
    # inputs that fit in L2 get a flush (a write of 2x L2) before every timed step; the flush sits
    # outside the per-step events, and the step time is then the sum of those per-step intervals
    flush = torch.empty(2 * l2 // 4, dtype=torch.int32, device=dev) if in_bytes < 2 * l2 else None
    for _ in range(max(3, args.warmup)):
        step(q, p)
    torch.cuda.synchronize(dev)
    assert int(status.item()) == 0, f"status flags {int(status.item())}"

    # ---- device-timed region
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk = Clocks(local)
    barrier(world)
    torch.cuda.synchronize(dev)
    clk.start()
    time.sleep(0.3)
    start.record(stream)
    for k in range(args.steps):
        if flush is not None:
            flush.fill_(k)
        step(q, p, evs[k])
    stop.record(stream)
    torch.cuda.synchronize(dev)
    clocks = clk.stop()
    barrier(world)
    if flush is None:
        ms = start.elapsed_time(stop)
        l2_note = f"inputs ({in_bytes / 1e9:.2f} GB) larger than L2, no flush"
    else:
        ms = sum(e[0].elapsed_time(e[2]) for e in evs)
        l2_note = (f"inputs ({in_bytes / 1e6:.1f} MB) fit in L2: {flush.numel() * 4 / 1e6:.0f} MB written "
                   f"before each step, outside the per-step events")
    ms = max_over_ranks(ms, world)
    t_draft = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    t_verify = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)

    esz = wl.p_logits.element_size()
    rows_per_step = t.n_nodes + t.n_draft
    bytes_verify = t.n_nodes * wl.vocab * esz
    bytes_draft = t.n_draft * wl.vocab * esz
    ms_step = ms / args.steps
    value = rows_per_step * world / (ms_step / 1e3)
    peak, peak_kind = _peaks()
    ach_v = bytes_verify / (t_verify / 1e3) / 1e9
    ach_d = bytes_draft / (t_draft / 1e3) / 1e9
    ach_all = (bytes_verify + bytes_draft) / (ms_step / 1e3) / 1e9
    # integer-multiply roof: 18 wide 32x32->64 multiplies per Philox4x32-10 block (rounds 1-2 of a
    # row share two products) = 4.5 per token; the multiply pipe retires 32 per SM per clock
    tok_verify = t.n_nodes * wl.vocab
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    clk = (clocks.get("sm_mhz") or 2070.0) * 1e6
    mul_peak = sms * WIDE_MULS_PER_SM_CLK * clk / 1e12
    muls_per_token = (2 * args.philox_rounds - 2) / 4  # rounds 1-2 hoisted: 2 R - 2 products per 4 tokens
    mul_ach = tok_verify * muls_per_token / (t_verify / 1e3) / 1e12
    traffic = None
    if args.workload == "zipf_k8" and args.n_seq is None:
        if args.top_k == 0:
            traffic = _traffic("verify")
        elif args.top_k == 50 and args.top_p == 1.0:
            traffic = _traffic("verify", TRUNC_TRAFFIC_FILE)
    philox_tok_s = philox_only_rate(dev) if rank == 0 else None
    emitted = float(vout["n_emitted"].sum().item())

    # ---- end to end through host buffers: every step copies its q and p logits from pinned host
    # memory (copy stream, two device buffers used in turn) and reads its emitted tokens and score
    # sums back.  The draft kernel waits only for q, the verify kernel for p, and the next step's
    # copies overlap this step's kernels.
    e2e = None
    if args.e2e_steps > 0:
        hq = torch.empty(q.shape, dtype=q.dtype, pin_memory=True)
        hp = torch.empty(p.shape, dtype=p.dtype, pin_memory=True)
        hq.copy_(q)
        hp.copy_(p)
        h_em = torch.empty(vout["emitted"].shape, dtype=torch.int32, pin_memory=True)
        h_ne = torch.empty(t.n_seq, dtype=torch.int32, pin_memory=True)
        h_ss = torch.empty(t.n_seq, dtype=torch.float64, pin_memory=True)
        bufs = [(torch.empty_like(q), torch.empty_like(p)) for _ in range(2)]
        copy_stream = torch.cuda.Stream(dev)
        freed = [torch.cuda.Event() for _ in range(2)]
        for f in freed:
            f.record(stream)

        def e2e_step(k):
            dq, dp2 = bufs[k & 1]
            ev_q, ev_p = torch.cuda.Event(), torch.cuda.Event()
            copy_stream.wait_event(freed[k & 1])  # the kernels of step k-2 are done with this buffer
            with torch.cuda.stream(copy_stream):
                dq.copy_(hq, non_blocking=True)
                ev_q.record(copy_stream)
                dp2.copy_(hp, non_blocking=True)
                ev_p.record(copy_stream)
            stream.wait_event(ev_q)
            draft(dq)
            stream.wait_event(ev_p)
            verify(dp2)
            freed[k & 1].record(stream)
            h_em.copy_(vout["emitted"], non_blocking=True)
            h_ne.copy_(vout["n_emitted"], non_blocking=True)
            h_ss.copy_(vout["score_sum"], non_blocking=True)

        e2e_step(0)
        torch.cuda.synchronize(dev)
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        copy_stream.wait_event(e0)
        for k in range(args.e2e_steps):
            e2e_step(k)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        e_ms = max_over_ranks(e0.elapsed_time(e1) / args.e2e_steps, world)
        e2e = {"value": rows_per_step * world / (e_ms / 1e3), "unit": "rows/s",
               "h2d_bytes_per_step": int(hq.numel() * esz + hp.numel() * esz),
               "d2h_bytes_per_step": int(h_em.numel() * 4 + h_ne.numel() * 4 + h_ss.numel() * 8),
               "ms_per_step": e_ms,
               "pipeline": "q and p copies on a copy stream, two device buffers; kernels wait per input"}
        del hq, hp, bufs

    cpu = None
    parity = None
    if rank == 0 and not args.no_cpu_baseline:
        import oracle
        # a step small enough for the CPU budget (the bench workload: ~7 s on 16 cores) is run whole,
        # once untimed and once timed, and its lists and winners are compared with the GPU's
        whole = args.top_k == 0 and (t.n_draft + t.n_nodes) <= 6000
        keep = {} if whole else None
        if whole:
            run, nd, nn, cores = oracle_sample(wl, t.n_draft, t.n_nodes, keep=keep)
        else:
            run, nd, nn, cores = oracle_sample(wl, 8, 8, top_k=args.top_k, top_p=args.top_p)
        dt = run()
        reps = max(1, int(args.cpu_seconds / max(dt, 1e-3)))
        tot = sum(run() for _ in range(reps))
        # one thread, on a small sample with the step's mix of draft and target rows
        n1d = max(1, round(16 * t.n_draft / (t.n_draft + t.n_nodes)))
        run1, nd1, nn1, _ = oracle_sample(wl, n1d, 16 - n1d, seed=1, top_k=args.top_k, top_p=args.top_p)
        oracle.set_threads(1)
        tot1 = run1()
        oracle.set_threads(cores)
        what = "every row of the step" if whole else "a sample of the step's rows"
        cpu = {"value": reps * (nd + nn) / tot, "unit": "rows/s", "cores": cores, "kind": "oracle",
               "sample": f"{what}: {nd} draft + {nn} target rows, x{reps} timed pass(es) after one untimed, "
                         f"{tot:.1f} s on {cores} threads",
               "single_thread_value": (nd1 + nn1) / tot1,
               "single_thread_sample": f"{nd1} draft + {nn1} target rows on 1 thread",
               "cpu_model": cpu_model(), "nproc": os.cpu_count()}
        if whole:
            parity = step_parity(wl, keep, dout, vout)

    # ---- the same step with the Philox4x32-7 keyed source (libpps_r7.so): a second number beside
    # the default's, with every row compared with the oracle at 7 rounds
    mean_acc = float(vout["accept_len"].float().mean().item())
    philox7 = None
    want7 = (args.workload == "zipf_k8" and args.n_seq is None and args.top_k == 0 and args.philox_rounds == 10
             and not args.no_philox7 and flush is None)
    if want7 and not os.path.exists(pps.library_path(7)):
        philox7 = {"unavailable": "libpps_r7.so was not built (build() makes both libraries)"}
    elif want7:
        pps.use_library(7)
        for _ in range(3):
            step(q, p)
        torch.cuda.synchronize(dev)
        evs7 = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
        s7, e7 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier(world)
        s7.record(stream)
        for k in range(args.steps):
            step(q, p, evs7[k])
        e7.record(stream)
        torch.cuda.synchronize(dev)
        ms7 = max_over_ranks(s7.elapsed_time(e7), world) / args.steps
        td7 = statistics.mean(e[0].elapsed_time(e[1]) for e in evs7)
        tv7 = statistics.mean(e[1].elapsed_time(e[2]) for e in evs7)
        ph7 = philox_only_rate(dev) if rank == 0 else None
        par7 = None
        if rank == 0 and not args.no_cpu_baseline and parity is not None:
            import oracle
            oracle.set_philox_rounds(7)
            keep7 = {}
            run7, _, _, _ = oracle_sample(wl, t.n_draft, t.n_nodes, keep=keep7)
            run7()
            par7 = step_parity(wl, keep7, dout, vout)
            oracle.set_philox_rounds(10)
        philox7 = {"keyed_source": "Philox4x32-7 (libpps_r7.so; an option beside the default)",
                   "value": rows_per_step * world / (ms7 / 1e3), "unit": "rows/s", "ms_per_step": ms7,
                   "roofline": {"bound": "hbm", "achieved": bytes_verify / (tv7 / 1e3) / 1e9, "peak": peak,
                                "unit": "GB/s", "frac": bytes_verify / (tv7 / 1e3) / 1e9 / peak, "ms": tv7,
                                "kernel": "race_kernel (pps_verify_tree)"},
                   "roofline_draft": {"frac": bytes_draft / (td7 / 1e3) / 1e9 / peak, "ms": td7},
                   "philox_only_tok_s": ph7,
                   "frac_of_philox_only": tok_verify / (tv7 / 1e3) / ph7 if ph7 else None,
                   "mean_accept_len": float(vout["accept_len"].float().mean().item()),
                   "parity": par7}
        pps.use_library(10)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if wl.dtype == torch.bfloat16 else "f32",
            "data": "synthetic (seeded Zipf-rank logits; no model, no dataset)",
            "config": {"workload": race_workload_name(args, wl),
                       "rows_per_step": rows_per_step, "l2": l2_note,
                       "parallelism": f"replicas x{world}"},
            "gb_per_s": ach_all, "emitted_tokens_per_s": emitted * world / (ms_step / 1e3),
            # the dominant kernel (verify, the larger of the two launches) against the measured HBM
            # copy bandwidth: algorithmic bytes = its rows x V x sizeof(logit), read once
            "roofline": {"bound": "hbm", "achieved": ach_v, "peak": peak, "unit": "GB/s", "frac": ach_v / peak,
                         "traffic": traffic, "peak_kind": f"{peak_kind} (MEASURED_PEAKS hbm_gbs)",
                         "kernel": ("trunc_kernel (pps_verify_tree_trunc)" if args.top_k > 0
                                    else "race_kernel (pps_verify_tree)"),
                         "ms": t_verify, "algorithmic_bytes": bytes_verify,
                         "bytes_per_row": wl.vocab * esz, "rows": t.n_nodes},
            "roofline_draft": {"bound": "hbm", "achieved": ach_d, "peak": peak, "unit": "GB/s",
                               "frac": ach_d / peak, "ms": t_draft, "algorithmic_bytes": bytes_draft,
                               "rows": t.n_draft},
            "roofline_step": {"achieved": ach_all, "frac": ach_all / peak, "unit": "GB/s",
                              "algorithmic_bytes": bytes_verify + bytes_draft},
            # the keyed source's own ceiling: Philox4x32-10 multiplies on the multiply pipe.  The
            # pipe rate is derived from ncu counters (not measured by the driver); the Philox-only
            # token rate is measured live by the library's self-test
            "roofline_alu": {"bound": "alu", "achieved": mul_ach, "peak": mul_peak, "unit": "T wide-mul/s",
                             "frac": mul_ach / mul_peak,
                             "peak_kind": f"derived, not measured: {sms} SMs x {WIDE_MULS_PER_SM_CLK} "
                                          f"32x32->64 multiplies/clk x {clk / 1e6:.0f} MHz (median sampled SM clock)",
                             "work": f"{muls_per_token} wide multiplies per token x {tok_verify} tokens",
                             "tok_s": tok_verify / (t_verify / 1e3), "philox_only_tok_s": philox_tok_s,
                             "frac_of_philox_only": (tok_verify / (t_verify / 1e3) / philox_tok_s
                                                     if philox_tok_s else None)},
            "e2e": e2e, "cpu_baseline": cpu, "gpu_launches": 2 * args.steps, "clocks": clocks,
            "mean_accept_len": mean_acc,
            "parity": parity,
            "keyed_source": f"Philox4x32-{args.philox_rounds}",
            "philox7": philox7,
        }
        print(json.dumps(line))


def step_parity(wl, keep, dout, vout):
    """The GPU step's lists, winners and accept lengths against the oracle's on every row of the
    step: flips (allowed only where the oracle's key gap is below 1e-6), mismatches (anything
    else: must be 0), the mean accept length of the oracle's own walk, and the depth-0 acceptance
    against the closed form of the IID list (App. B, Thm B.2: exact for multi-arrival lists, a
    lower bound for the DISTINCT lists timed here)."""
    import oracle
    from oracle import closed_forms as cf
    t = wl.tree
    od = keep["draft"]
    win_o, wd_o, _, mg_o = keep["target"]
    tok_g = dout["tok"].cpu().numpy()
    win_g = vout["winner"].cpu().numpy()
    d_bad = np.nonzero(np.any(tok_g != od["tok"], axis=1))[0]
    n_bad = np.nonzero(win_g != win_o)[0]
    d_flip = int(np.sum(od["min_gap"][d_bad] < 1e-6))
    n_flip = int(np.sum(mg_o[n_bad] < 1e-6))
    ow = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, od["tok"], od["ndist"], t.child_node, win_o, wd_o)
    acc_g = vout["accept_len"].cpu().numpy()
    roots = t.seq_off[:-1].astype(np.int64)
    droots = t.node_draft_row[roots].astype(np.int64)
    P = wl.p_logits[torch.as_tensor(roots, device=wl.p_logits.device)].double().cpu().numpy()
    Q = wl.q_logits[torch.as_tensor(droots, device=wl.q_logits.device)].double().cpu().numpy()
    T = float(np.float32(wl.temperature))
    pr = np.array([cf.accept_iid_full(cf.softmax(P[s], T), cf.softmax(Q[s], T), int(t.row_k[droots[s]]))
                   for s in range(t.n_seq)])
    return {"rows_compared": f"{t.n_draft} draft + {t.n_nodes} target (every row of the step)",
            "draft_flips": d_flip, "winner_flips": n_flip,
            "mismatches": int(len(d_bad) - d_flip + len(n_bad) - n_flip),
            "accept_len_equal_to_oracle": bool(np.array_equal(acc_g, ow["accept_len"])),
            "mean_accept_len": {"gpu": float(acc_g.mean()), "oracle": float(ow["accept_len"].mean())},
            "depth0_accept": {"gpu": float(np.mean(acc_g >= 1)), "oracle": float(np.mean(ow["accept_len"] >= 1)),
                              "closed_form_iid": float(pr.mean()),
                              "binomial_sd": float(np.sqrt(np.sum(pr * (1 - pr))) / t.n_seq),
                              "note": "IID closed form: exact for multi-arrival lists, a lower bound for "
                                      "the DISTINCT lists of this step"}}


def run_detector(args, rank, world, dev):
    """Detector pass (pps_wm_detect: Aaronson scores, per-segment sums and exact Gamma-tail
    log p-values) over n_tokens (token, key, label, position) tuples in segments (texts) of
    128 with one watermark key per text: the
    first half watermarked (race winners of fresh contexts, drawn by pps_verify_tree over
    N(0, 3^2) logits of 256 tokens), the second half uniform-random tokens (the null)."""
    from paper_2609_21858_gb300 import pps
    n = args.n_tokens - args.n_tokens % 256
    half = n // 2
    g = torch.Generator(device=dev)
    g.manual_seed(4)
    # one watermark key per text (segment of 128 tokens); labels and positions per token
    key = torch.randint(-2 ** 62, 2 ** 62, (n // 128,), generator=g, device=dev, dtype=torch.int64).repeat_interleave(128)
    ctx = torch.randint(-2 ** 62, 2 ** 62, (n,), generator=g, device=dev, dtype=torch.int64)
    pos = torch.randint(0, 2 ** 30, (n,), generator=g, device=dev, dtype=torch.int32)
    tok = torch.randint(0, 128256, (n,), generator=g, device=dev, dtype=torch.int32)
    # watermarked half: each context's token is the target race winner (one-node trees)
    Vw = 256
    logits = torch.randn(half, Vw, generator=g, device=dev).mul_(3.0).to(torch.bfloat16)
    ar = torch.arange(half + 1, device=dev, dtype=torch.int32)
    none = torch.full((half,), -1, device=dev, dtype=torch.int32)
    v = pps.verify_tree(logits, key[:half], ctx[:half], pos[:half], 1, ar, none,
                        torch.full((1, 1), -1, device=dev, dtype=torch.int32),
                        torch.zeros(1, device=dev, dtype=torch.int32),
                        torch.full((1, 1), -1, device=dev, dtype=torch.int32))
    tok[:half] = v["winner"]
    del logits, v
    seg = torch.arange(0, n + 1, 128, device=dev, dtype=torch.int64)
    stream = torch.cuda.current_stream(dev)
    for _ in range(max(3, args.warmup)):
        sc, sums, logp = pps.wm_detect(tok, key, ctx, pos, seg, want_scores=False, stream=stream)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk = Clocks(dev.index or 0)
    barrier(world)
    clk.start()
    time.sleep(0.3)
    e0.record(stream)
    for _ in range(args.steps):
        sc, sums, logp = pps.wm_detect(tok, key, ctx, pos, seg, want_scores=False, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    clocks = clk.stop()
    ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, world)
    # the score kernel alone (scores and segment sums, no p-values): the pass's dominant kernel
    barrier(world)
    e0.record(stream)
    for _ in range(args.steps):
        pps.wm_detect(tok, key, ctx, pos, seg, want_scores=False, want_logp=False, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    ms_score = max_over_ranks(e0.elapsed_time(e1) / args.steps, world)
    n_seg = seg.numel() - 1
    bytes_in = n * (4 + 8 + 8 + 4) + seg.numel() * 8
    bytes_out = n_seg * 16
    peak, peak_kind = _peaks()
    gbs = (bytes_in + bytes_out) / (ms / 1e3) / 1e9
    gbs_score = (bytes_in + n_seg * 8) / (ms_score / 1e3) / 1e9
    lp = logp.cpu().numpy()
    wm, null = lp[: n_seg // 2], lp[n_seg // 2:]
    alpha = np.log(0.01)
    if rank == 0:
        print(json.dumps({
            "metric": "watermark detector pass with p-values (tokens/s)", "value": n * world / (ms / 1e3),
            "unit": "tokens/s", "n_gpus": world, "steps": args.steps, "warmup": max(3, args.warmup),
            "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": f"detector: {n} tuples in segments of 128, half watermarked, Aaronson "
                                   f"scores, exact Gamma-tail p-values",
                       "l2": f"inputs ({bytes_in / 1e6:.0f} MB) larger than L2, no flush"},
            "roofline": {"bound": "hbm", "achieved": gbs_score, "peak": peak, "unit": "GB/s",
                         "frac": gbs_score / peak, "traffic": None, "peak_kind": peak_kind,
                         "kernel": "wm_score_kernel (scores and segment sums, incl. the sums' memset)",
                         "ms": ms_score, "algorithmic_bytes": bytes_in + n_seg * 8},
            "pass": {"achieved_gbs": gbs, "frac_hbm": gbs / peak, "algorithmic_bytes": bytes_in + bytes_out,
                     "pvalue_ms": ms - ms_score},
            "detection": {"tpr_at_1pct_fpr": float(np.mean(wm <= alpha)), "fpr_null": float(np.mean(null <= alpha)),
                          "anlppt_watermarked": float(np.mean(-wm / 128.0)),
                          "anlppt_null": float(np.mean(-null / 128.0)), "segments": int(n_seg)},
            "gpu_launches": 2 * args.steps, "clocks": clocks, "keyed_source": f"Philox4x32-{args.philox_rounds}",
        }))


def run_dynamic(args, rank, world, dev):
    """The dynamic IID draft tree (the paper's multi-draft tree: every context draws its
    multiplicity nu(c) of i.i.d. samples, K paths per depth): per step gamma pps_draft_list (IID)
    + pps_tree_expand calls, then pps_verify_tree over every node slot.  B=64, V=128256, K=8,
    gamma=5 (fixed capacity 41 node slots and 33 draft rows per sequence), bf16 logits: target
    rows as zipf_k8, drafts = the node's target row + N(0,1) (the drafter's outputs are inputs)."""
    from paper_2609_21858_gb300 import pps, synth, tree
    n_seq, V, K, gamma = args.n_seq or 64, 128256, 8, 5
    g = torch.Generator(device=dev)
    g.manual_seed(2)
    b = tree.TreeBuilder(n_seq, K, gamma, dev)
    p = synth._zipf(g, b.n_nodes, V, 1.0, True, dev).to(torch.bfloat16)
    N1 = 1 + K * gamma
    q = []
    for d in range(gamma):
        off = 0 if d == 0 else 1 + (d - 1) * K
        w = 1 if d == 0 else K
        slots = (torch.arange(n_seq, device=dev)[:, None] * N1 + off + torch.arange(w, device=dev)[None, :]).ravel()
        q.append((p[slots].float() + torch.randn(slots.numel(), V, generator=g, device=dev)).to(torch.bfloat16))
    rk = torch.as_tensor(synth.splitmix64_stream(20, 2 * n_seq).view(np.int64), device=dev)
    root_key, root_ctx = rk[:n_seq], rk[n_seq:]
    root_pos = torch.arange(n_seq, dtype=torch.int32, device=dev) * 0 + 100
    ws_v = pps.workspace(b.n_nodes, n_seq, dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    W = gamma + 1
    vout = dict(winner=torch.empty(b.n_nodes, dtype=torch.int32, device=dev),
                word=torch.empty(b.n_nodes, dtype=torch.int32, device=dev),
                accept_len=torch.empty(n_seq, dtype=torch.int32, device=dev),
                n_emitted=torch.empty(n_seq, dtype=torch.int32, device=dev),
                emitted=torch.empty(n_seq, W, dtype=torch.int32, device=dev),
                score=torch.empty(n_seq, W, dtype=torch.float32, device=dev),
                score_sum=torch.empty(n_seq, dtype=torch.float64, device=dev))
    def step():
        b.run(root_key, root_ctx, root_pos, lambda d, *_: q[d])
        b.verify(p, ws=ws_v, out=vout, status=status)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    assert int(status.item()) == 0, f"status flags {int(status.item())}"
    run = step if args.eager else graph_of(step, dev).replay
    barrier(world)
    ms, clocks = timed_replays(run, args.steps, dev, Clocks(dev.index or 0))
    ms = max_over_ranks(ms, world)
    rows = b.n_draft + b.n_nodes
    nbytes = rows * V * 2
    peak, peak_kind = _peaks()
    gbs = nbytes / (ms / 1e3) / 1e9
    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": rows * world / (ms / 1e3), "unit": "rows/s", "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded Zipf-rank logits; no model, no dataset)",
            "config": {"workload": f"dynamic IID tree: B={n_seq}, V={V}, K={K}, gamma={gamma}, "
                                   f"{b.n_nodes} node slots + {b.n_draft} draft rows per step",
                       "rows_per_step": rows, "l2": f"inputs ({nbytes / 1e9:.2f} GB) larger than L2, no flush",
                       "parallelism": f"replicas x{world}",
                       "launch": "eager" if args.eager else "CUDA graph of the step's library calls"},
            "gb_per_s": gbs,
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak,
                         "traffic": None, "peak_kind": peak_kind, "algorithmic_bytes": nbytes},
            "gpu_launches": args.steps * (2 * gamma + 1), "clocks": clocks,
            "keyed_source": f"Philox4x32-{args.philox_rounds}",
            "mean_accept_len": float(vout["accept_len"].float().mean().item()),
            "mean_draft_nodes_per_seq": float((b.row_k[:b.n_draft] > 0).sum().item()) / n_seq,
        }))


def graph_of(fn, dev):
    """Capture fn() (library calls on the current stream) into a CUDA graph, after warm-up
    runs on the capture's side stream."""
    side = torch.cuda.Stream(dev)
    side.wait_stream(torch.cuda.current_stream(dev))
    with torch.cuda.stream(side):
        for _ in range(3):
            fn()
    torch.cuda.current_stream(dev).wait_stream(side)
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    torch.cuda.synchronize(dev)
    return g


def timed_replays(fn, steps, dev, clk=None):
    """Mean device time of `steps` calls of fn on the current stream (CUDA events)."""
    stream = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    if clk is not None:
        clk.start()
        time.sleep(0.3)
    e0.record(stream)
    for _ in range(steps):
        fn()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    clocks = clk.stop() if clk is not None else None
    return e0.elapsed_time(e1) / steps, clocks


def run_hetero(args, rank, world, dev):
    """Non-identical proposals (the augmented race on V x [B], B = 8 draft models): per step
    gamma x (pps_draft_hetero over the n_seq x B proposal rows + pps_hetero_expand), then
    pps_verify_tree over every node slot of the merged chains.  n_seq=64, V=128256, B=8,
    gamma=5 (41 node slots and 40 proposal rows per sequence), bf16 logits: target rows as
    zipf_k8; proposal b's rows = the target row of its static slot + N(0, (0.5 + 0.25 b)^2)
    (the drafters' outputs are inputs)."""
    from paper_2609_21858_gb300 import pps, synth, tree
    n_seq, V, B, gamma = args.n_seq or 64, 128256, 8, 5
    g = torch.Generator(device=dev)
    g.manual_seed(3)
    b = tree.HeteroTreeBuilder(n_seq, B, gamma, dev)
    p = synth._zipf(g, b.n_nodes, V, 1.0, True, dev).to(torch.bfloat16)
    N1 = 1 + B * gamma
    sig = (0.5 + 0.25 * torch.arange(B, device=dev, dtype=torch.float32)).repeat(n_seq)[:, None]
    q = []
    for d in range(gamma):
        # row (s, b) of depth d reads node (s, d, b)'s target row (the root at depth 0)
        off = 0 if d == 0 else 1 + (d - 1) * B
        w = torch.arange(B, device=dev) if d > 0 else torch.zeros(B, dtype=torch.long, device=dev)
        slots = (torch.arange(n_seq, device=dev)[:, None] * N1 + off + w[None, :]).ravel()
        q.append((p[slots].float() + sig * torch.randn(slots.numel(), V, generator=g, device=dev))
                 .to(torch.bfloat16))
    rk = torch.as_tensor(synth.splitmix64_stream(30, 2 * n_seq).view(np.int64), device=dev)
    root_key, root_ctx = rk[:n_seq], rk[n_seq:]
    root_pos = torch.full((n_seq,), 100, dtype=torch.int32, device=dev)
    ws_v = pps.workspace(b.n_nodes, n_seq, dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    W = gamma + 1
    vout = dict(winner=torch.empty(b.n_nodes, dtype=torch.int32, device=dev),
                word=torch.empty(b.n_nodes, dtype=torch.int32, device=dev),
                accept_len=torch.empty(n_seq, dtype=torch.int32, device=dev),
                n_emitted=torch.empty(n_seq, dtype=torch.int32, device=dev),
                emitted=torch.empty(n_seq, W, dtype=torch.int32, device=dev),
                score=torch.empty(n_seq, W, dtype=torch.float32, device=dev),
                score_sum=torch.empty(n_seq, dtype=torch.float64, device=dev))
    tk, tp = args.top_k, args.top_p

    def draft():
        b.run(root_key, root_ctx, root_pos, lambda d, *_: q[d], top_k=tk, top_p=tp)

    def verify():
        b.verify(p, ws=ws_v, out=vout, status=status, top_k=tk, top_p=tp)

    def step():
        draft()
        verify()

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    assert int(status.item()) == 0, f"status flags {int(status.item())}"
    if args.eager:
        run, run_d, run_v = step, draft, verify
    else:
        run, run_d, run_v = (graph_of(f, dev).replay for f in (step, draft, verify))
    barrier(world)
    ms, clocks = timed_replays(run, args.steps, dev, Clocks(dev.index or 0))
    ms = max_over_ranks(ms, world)
    # the two phases alone (the draft phase: gamma proposal-row races + expansions)
    t_draft, _ = timed_replays(run_d, args.steps, dev)
    t_verify, _ = timed_replays(run_v, args.steps, dev)
    n_prop = gamma * n_seq * B
    rows = n_prop + b.n_nodes
    nbytes = rows * V * 2
    peak, peak_kind = _peaks()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    hz = (clocks.get("sm_mhz") or 2070.0) * 1e6
    mul_peak = sms * WIDE_MULS_PER_SM_CLK * hz / 1e12
    tok_draft = n_prop * V
    muls_per_token = (2 * args.philox_rounds - 2) / 4
    mul_ach = tok_draft * muls_per_token / (t_draft / 1e3) / 1e12
    trunc = f", top-k {tk}, top-p {tp}" if tk > 0 else ""
    roof_alu = {"bound": "alu", "achieved": mul_ach, "peak": mul_peak, "unit": "T wide-mul/s",
                "frac": mul_ach / mul_peak,
                "peak_kind": f"derived, not measured: {sms} SMs x {WIDE_MULS_PER_SM_CLK} 32x32->64 "
                             f"multiplies/clk x {hz / 1e6:.0f} MHz (median sampled SM clock)",
                "work": f"{muls_per_token} wide multiplies per token x {tok_draft} tokens"}
    gbs_d = n_prop * V * 2 / (t_draft / 1e3) / 1e9
    kern = "trunc_kernel" if tk > 0 else "race_kernel"
    roof = {"bound": "hbm", "achieved": gbs_d, "peak": peak, "unit": "GB/s", "frac": gbs_d / peak,
            "traffic": None, "kernel": f"{kern}, proposal rows (pps_draft_hetero{'_trunc' if tk > 0 else ''}) "
                                       f"incl. the expansions",
            "ms": t_draft, "peak_kind": peak_kind, "algorithmic_bytes": n_prop * V * 2}
    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": rows * world / (ms / 1e3), "unit": "rows/s", "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded Zipf-rank logits; no model, no dataset)",
            "config": {"workload": f"non-identical proposals: n_seq={n_seq}, V={V}, B={B} proposals, "
                                   f"gamma={gamma}, {n_prop} proposal rows + {b.n_nodes} node slots per step{trunc}",
                       "rows_per_step": rows, "l2": f"inputs ({nbytes / 1e9:.2f} GB) larger than L2, no flush",
                       "parallelism": f"replicas x{world}",
                       "launch": "eager" if args.eager else "CUDA graph of the step's library calls"},
            "gb_per_s": nbytes / (ms / 1e3) / 1e9,
            "roofline": roof,
            "roofline_alu": None if tk > 0 else roof_alu,
            "roofline_verify": {"bound": "hbm", "achieved": b.n_nodes * V * 2 / (t_verify / 1e3) / 1e9,
                                "peak": peak, "peak_kind": peak_kind, "ms": t_verify},
            "gpu_launches": args.steps * (2 * gamma + 1), "clocks": clocks,
            "keyed_source": f"Philox4x32-{args.philox_rounds}",
            "mean_accept_len": float(vout["accept_len"].float().mean().item()),
            "mean_nodes_per_seq": float((b.node_ctx != 0).sum().item()) / n_seq,
        }))


def _peak_tflops():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured"
    except Exception:
        return 1900.0, 1700.0, "fallback"


def run_lmhead(args, rank, world, dev):
    """The race fused into the LM head (pps_lmhead_draft_list + pps_lmhead_verify_tree): the
    zipf_k8 tree of B=64 sequences (K=8, gamma=5), V=128256, target hidden size 4096 (2624 node
    rows), draft hidden size 2048 (2112 draft rows), bf16 operands whose products are Zipf-shaped
    logits (synth.lmhead_workload).  One step = the draft GEMM + race and the target GEMM + race +
    tree walk; no logits reach HBM.  The unfused step (pps_lmhead_logits twice, then
    pps_draft_list and pps_verify_tree on the fp32 logits) is timed beside it."""
    from paper_2609_21858_gb300 import pps, synth
    n_seq = args.n_seq or 64
    wl = synth.lmhead_workload(n_seq=n_seq, device=dev)
    t = wl.tree
    g = lambda x: torch.as_tensor(np.asarray(x)).to(dev).contiguous()
    rk, so, ndr, cn = g(t.row_k), g(t.seq_off), g(t.node_draft_row), g(t.child_node)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    wsd, wsv = pps.lmhead_workspace(t.n_draft, 0, dev), pps.lmhead_workspace(t.n_nodes, t.n_seq, dev)
    stream = torch.cuda.current_stream(dev)
    dout = pps.lmhead_draft_list(wl.hq, wl.wq, wl.draft_key, wl.draft_ctx, wl.draft_pos, t.K, row_k=rk, ws=wsd,
                                 status=status, keys=False, samples=False)
    vout = pps.lmhead_verify_tree(wl.hp, wl.wp, wl.node_key, wl.node_ctx, wl.node_pos, t.gamma, so, ndr,
                                  dout["tok"], dout["ndist"], cn, ws=wsv, status=status)

    def step(hq=wl.hq, hp=wl.hp, ev=None):
        if ev is not None:
            ev[0].record(stream)
        pps.lmhead_draft_list(hq, wl.wq, wl.draft_key, wl.draft_ctx, wl.draft_pos, t.K, row_k=rk, ws=wsd,
                              status=status, out=dout, stream=stream)
        if ev is not None:
            ev[1].record(stream)
        pps.lmhead_verify_tree(hp, wl.wp, wl.node_key, wl.node_ctx, wl.node_pos, t.gamma, so, ndr, dout["tok"],
                               dout["ndist"], cn, ws=wsv, status=status, out=vout, stream=stream)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    assert int(status.item()) == 0, f"status flags {int(status.item())}"
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk = Clocks(dev.index or 0)
    barrier(world)
    torch.cuda.synchronize(dev)
    clk.start()
    time.sleep(0.3)
    e0.record(stream)
    for k in range(args.steps):
        step(ev=evs[k])
    e1.record(stream)
    torch.cuda.synchronize(dev)
    clocks = clk.stop()
    ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, world)
    t_d = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    t_v = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    V, dt_, dd_ = wl.vocab, wl.hp.shape[1], wl.hq.shape[1]
    fl_v, fl_d = 2.0 * t.n_nodes * V * dt_, 2.0 * t.n_draft * V * dd_
    peak, peak_sus, peak_kind = _peak_tflops()
    # the unfused step: the same GEMMs writing fp32 logits, then the streaming race
    lq = torch.empty(t.n_draft, V, device=dev)
    lp = torch.empty(t.n_nodes, V, device=dev)
    ud = pps.draft_list(lq, wl.draft_key, wl.draft_ctx, wl.draft_pos, t.K, row_k=rk)
    uv = pps.verify_tree(lp, wl.node_key, wl.node_ctx, wl.node_pos, t.gamma, so, ndr, ud["tok"], ud["ndist"], cn)

    def unfused():
        pps.lmhead_logits(wl.hq, wl.wq, out=lq, stream=stream)
        pps.draft_list(lq, wl.draft_key, wl.draft_ctx, wl.draft_pos, t.K, row_k=rk, out=ud, stream=stream)
        pps.lmhead_logits(wl.hp, wl.wp, out=lp, stream=stream)
        pps.verify_tree(lp, wl.node_key, wl.node_ctx, wl.node_pos, t.gamma, so, ndr, ud["tok"], ud["ndist"], cn,
                        out=uv, stream=stream)

    for _ in range(2):
        unfused()
    ms_unfused, _ = timed_replays(unfused, max(3, args.steps // 2), dev)
    same = bool(torch.equal(uv["emitted"], vout["emitted"]) and torch.equal(ud["tok"], dout["tok"]))
    del lq, lp
    # end to end: the step's hidden states come from pinned host memory (the LM-head weights stay
    # resident, as a serving engine keeps them), its emitted tokens and score sums go back
    e2e = None
    if args.e2e_steps > 0:
        hq_h = torch.empty(wl.hq.shape, dtype=wl.hq.dtype, pin_memory=True)
        hp_h = torch.empty(wl.hp.shape, dtype=wl.hp.dtype, pin_memory=True)
        hq_h.copy_(wl.hq)
        hp_h.copy_(wl.hp)
        hq_d, hp_d = torch.empty_like(wl.hq), torch.empty_like(wl.hp)
        em_h = torch.empty(vout["emitted"].shape, dtype=torch.int32, pin_memory=True)
        ss_h = torch.empty(t.n_seq, dtype=torch.float64, pin_memory=True)

        def e2e_step():
            hq_d.copy_(hq_h, non_blocking=True)
            hp_d.copy_(hp_h, non_blocking=True)
            step(hq_d, hp_d)
            em_h.copy_(vout["emitted"], non_blocking=True)
            ss_h.copy_(vout["score_sum"], non_blocking=True)

        e2e_step()
        torch.cuda.synchronize(dev)
        e_ms, _ = timed_replays(e2e_step, args.e2e_steps, dev)
        e_ms = max_over_ranks(e_ms, world)
        rows = t.n_nodes + t.n_draft
        e2e = {"value": rows * world / (e_ms / 1e3), "unit": "rows/s",
               "h2d_bytes_per_step": int((hq_h.numel() + hp_h.numel()) * 2),
               "d2h_bytes_per_step": int(em_h.numel() * 4 + ss_h.numel() * 8), "ms_per_step": e_ms}
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = lmhead_oracle_sample(wl, args.cpu_seconds)
    if rank == 0:
        rows = t.n_nodes + t.n_draft
        ach = (fl_v + fl_d) / (ms / 1e3) / 1e12
        print(json.dumps({
            "metric": METRIC, "value": rows * world / (ms / 1e3), "unit": "rows/s", "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded hidden states and LM-head weights with Zipf-shaped products; no model)",
            "config": {"workload": f"lmhead: B={t.n_seq}, V={V}, K={t.K}, gamma={t.gamma}, d={dt_} target / {dd_} "
                                   f"draft, {t.n_nodes} node rows + {t.n_draft} draft rows per step, race fused "
                                   f"into the LM-head GEMM",
                       "rows_per_step": rows, "l2": f"weights ({(wl.wp.numel() + wl.wq.numel()) * 2 / 1e9:.2f} GB) "
                                                   f"larger than L2, no flush",
                       "parallelism": f"replicas x{world}"},
            "roofline": {"bound": "tensor", "achieved": ach, "peak": peak, "unit": "TFLOP/s", "frac": ach / peak,
                         "traffic": None, "peak_kind": f"{peak_kind} (MEASURED_PEAKS bf16_tflops, cuBLAS burst)",
                         "kernel": "lmhead_kernel<RaceEpi> (both launches of the step, with their finishing kernels)",
                         "ms": ms, "flops": fl_v + fl_d, "frac_of_sustained": ach / peak_sus},
            "launches": {"draft_ms": t_d, "draft_tflops": fl_d / (t_d / 1e3) / 1e12,
                         "verify_ms": t_v, "verify_tflops": fl_v / (t_v / 1e3) / 1e12},
            "unfused": {"ms_per_step": ms_unfused, "speedup_of_fusion": ms_unfused / ms,
                        "same_outputs": same,
                        "logits_bytes_avoided": int((t.n_nodes + t.n_draft) * V * 4 * 2)},
            "e2e": e2e, "cpu_baseline": cpu, "gpu_launches": 4 * args.steps, "clocks": clocks,
            "keyed_source": f"Philox4x32-{args.philox_rounds}",
            "mean_accept_len": float(vout["accept_len"].float().mean().item()),
        }))


def lmhead_oracle_sample(wl, seconds: float):
    """The oracle (fp64 LM head, then its race) on a bounded sample of the step's rows."""
    import oracle
    t = wl.tree
    cores = oracle.set_threads(0)
    rng = np.random.default_rng(0)
    nr = np.sort(rng.choice(t.n_nodes, 16, replace=False))
    dr = np.sort(rng.choice(t.n_draft, 13, replace=False))
    hp = wl.hp[torch.as_tensor(nr, device=wl.hp.device)].float().cpu().numpy()
    hq = wl.hq[torch.as_tensor(dr, device=wl.hq.device)].float().cpu().numpy()
    wp, wq = wl.wp.float().cpu().numpy(), wl.wq.float().cpu().numpy()
    from paper_2609_21858_gb300 import synth
    ids_n = (synth.u64(wl.node_key)[nr], synth.u64(wl.node_ctx)[nr], synth.u32(wl.node_pos)[nr])
    ids_d = (synth.u64(wl.draft_key)[dr], synth.u64(wl.draft_ctx)[dr], synth.u32(wl.draft_pos)[dr])

    def run():
        t0 = time.perf_counter()
        lq = oracle.lmhead_logits(hq, wq).astype(np.float32)
        oracle.draft_rows(lq, *ids_d, t.K, row_k=t.row_k[dr])
        lp = oracle.lmhead_logits(hp, wp).astype(np.float32)
        oracle.target_rows(lp, *ids_n)
        return time.perf_counter() - t0

    dt = run()
    reps = max(1, int(seconds / max(dt, 1e-3)))
    tot = sum(run() for _ in range(reps))
    return {"value": reps * (len(nr) + len(dr)) / tot, "unit": "rows/s", "cores": cores, "kind": "oracle",
            "sample": f"{len(dr)} draft + {len(nr)} target rows (fp64 LM head + race), x{reps} after one untimed, "
                      f"{tot:.1f} s on {cores} threads", "cpu_model": cpu_model(), "nproc": os.cpu_count()}


def run_reference(args, world):
    """The CPU oracle on a bounded sample per step, on this host's cores."""
    from paper_2609_21858_gb300 import synth
    if args.workload == "lmhead":
        wl = synth.lmhead_workload(device="cuda" if torch.cuda.is_available() else "cpu")
        cpu = lmhead_oracle_sample(wl, 2.0 * args.steps)
        t = wl.tree
        print(json.dumps({
            "impl": "reference", "metric": METRIC, "value": cpu["value"], "unit": "rows/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"lmhead: B={t.n_seq}, V={wl.vocab}, K={t.K}, gamma={t.gamma}",
                       "parallelism": f"replicas x{world}"},
            "cpu_baseline": cpu,
            "e2e": {"value": cpu["value"], "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))
        return
    wl = synth.make_workload(args.workload, device="cuda" if torch.cuda.is_available() else "cpu",
                             K_sweep=args.k if args.workload == "ksweep" else None)
    t = wl.tree
    # a sixteenth of the step per timed step, with the step's mix of draft and target rows (at
    # least as many rows as host threads)
    frac = max(1.0 / 16.0, 32.0 / (t.n_draft + t.n_nodes))
    run, nd, nn, cores = oracle_sample(wl, max(1, round(t.n_draft * frac)), max(1, round(t.n_nodes * frac)),
                                       top_k=args.top_k, top_p=args.top_p)
    for _ in range(max(1, min(args.warmup, 2))):
        run()
    times = [run() for _ in range(args.steps)]
    tot = sum(times)
    value = args.steps * (nd + nn) / tot
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": race_workload_name(args, wl), "rows_per_step": nd + nn,
                   "parallelism": f"replicas x{world}"},
        "cpu_baseline": {"value": value, "unit": "rows/s", "cores": cores, "kind": "oracle",
                         "sample": f"{nd} draft + {nn} target rows per step", "cpu_model": cpu_model(),
                         "nproc": os.cpu_count()},
        "e2e": {"value": value, "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


if __name__ == "__main__":
    main()
