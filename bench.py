#!/usr/bin/env python
"""Benchmark of the trie-automaton hot path on GB300.

One step = one schema through the whole path: mask compile for every trie
node (k_mask_probe | k_mask_fill_beside -> k_mask_scatter) and then the
batched decode loop: step 0 masks its logits (k_apply_vec), every later step
advances the states by the previous step's greedy tokens and masks its own
logits in one launch (k_advance_apply_vec), and a last advance (k_advance)
follows. The greedy choice itself is the
caller's sampler, not part of the path: the tokens are computed once before
timing and replayed. The workload is K = 10,000 ICD-style codes with a
152,064-token byte vocabulary, batch 256, 16 decode steps, bf16 logits.

value     (node, token) pairs per second, N * V per step over the device time
          of the step, inputs resident in HBM (one CUDA graph per step).
e2e       the same pairs/s through the C ABI from host buffers: the trie
          built from host strings, logits and tokens copied from pinned host
          memory, the states read back every decode step.
roofline  the dominant kernel of the step (mask application), algorithmic
          bytes per launch over its CUDA-event duration inside the timed
          replay; roofline_compile gives the same for the mask compile.

`--impl reference` times the CPU oracle (plain C, OpenMP) on the same
workload instead. With torchrun (N > 1) every rank runs its own replica
(weak scaling; the path needs no exchange between GPUs).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "mask-compile ms & (node,token) pairs/s; batch-256 mask-apply GB/s vs HBM peak"
UNIT = "pairs/s"
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=1000)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    p.add_argument("--config", type=int, default=3, choices=[1, 2, 3, 4])
    p.add_argument("--e2e-steps", type=int, default=10)
    p.add_argument("--cpu-seconds", type=float, default=10.0,
                   help="time budget of the CPU-oracle baseline sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-dynamic", action="store_true", help="skip the dynamic per-query-set measurement")
    p.add_argument("--no-graph", action="store_true", help="run the steps eagerly instead of as CUDA graphs")
    p.add_argument("--profile", choices=["compile", "pairwise", "lists", "listdecode", "lazy", "step"],
                   help="run one part of the path alone (for profilers) and print its CUDA-event time "
                        "instead of the JSON line")
    p.add_argument("--requests", type=int, default=256, help="--profile lists: requests of the forest")
    p.add_argument("--device-build", action="store_true", help="--profile lists: build the forest on the GPU")
    p.add_argument("--cache-rows", type=int, default=0, help="--profile lazy: row cache size")
    p.add_argument("--reps", type=int, default=5, help="--profile: repetitions")
    return p.parse_args()


def peaks() -> tuple[float, str]:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash(path: str | None = None) -> str:
    """Hash of kernels.cu (or `path`) without its // comments and blank lines:
    a traffic record stays valid across comment edits and lapses with any
    code change."""
    path = path or os.path.join(ROOT, "paper_2608_12574_gb300", "csrc", "kernels.cu")
    with open(path, "rb") as f:
        lines = [ln.split("//", 1)[0].rstrip() for ln in f.read().decode().splitlines()]
    return hashlib.sha256("\n".join(ln for ln in lines if ln.strip()).encode()).hexdigest()[:16]


def ncu_traffic(kernel: str, workload: str) -> float | None:
    """DRAM bytes per launch recorded by ncu for this kernel source, else None."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    if not os.path.exists(path):
        return None
    h = kernel_source_hash()
    for line in open(path):
        parts = line.split()
        if len(parts) == 4 and parts[0] == kernel and parts[1] == workload and parts[2] == h:
            return float(parts[3])
    return None


class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.proc = None
        self.uuid = uuid

    def __enter__(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "100"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        time.sleep(0.2)
        self.out = ""
        if self.proc:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self) -> dict:
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (getattr(self, "out", "") or "").splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                smax.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def compile_kernels(w, n_nodes: int, max_depth: int, num_sms: int) -> int:
    """Kernels one trie_compile_masks launches, by the library's rule: a mask
    of at most 32 MB of a trie whose search takes two threads per node (at
    most num_sms * 128 nodes, tokens and depth within 16 bytes, no repeated
    token string, so that every table slot holds one token's payload) is the
    fill and the search ORing its hits (2); otherwise the search, the fill and
    the scatter (3). (Two distinct strings whose 64-bit keys collide also
    take the 3-kernel form; that is not modelled.)"""
    import numpy as np
    vb, vo = np.asarray(w.vocab_bytes), np.asarray(w.vocab_offsets)
    lens = np.diff(vo)[: w.V - 1]  # token V - 1 is EOS: its bytes are ignored
    lmax = min(int(lens.max()) if lens.size else 0, max_depth)
    strings = [bytes(vb[vo[i]:vo[i + 1]]) for i in range(w.V - 1) if lens[i] > 0]
    pair = lmax <= 16 and 4 * n_nodes <= num_sms * 4 * 128 and len(set(strings)) == len(strings)
    mask_bytes = n_nodes * ((w.V + 31) // 32) * 4
    return 2 if pair and mask_bytes <= (32 << 20) else 3


def workload_config(w, n_nodes: int) -> dict:
    """The `config` object of the JSON line, the same in both arms: the
    workload and its sizes (N_chars = bytes of the distinct set strings, r =
    N / N_chars as in App. H.7) and how L2 reuse is ruled out."""
    from paper_2608_12574_gb300 import workloads as W
    n_chars = sum(len(x) for x in set(W.unpack(w.set_bytes, w.set_offsets)))
    elt = 2 if w.dtype == "bf16" else 4
    mask_bytes = n_nodes * ((w.V + 31) // 32) * 4
    return {"workload": w.name, "K": w.K, "V": w.V, "batch": w.batch, "decode_steps": w.steps,
            "N_nodes": n_nodes, "N_chars": n_chars, "r": round(n_nodes / max(1, n_chars), 4),
            "l2": f"inputs larger than L2: logits {w.steps * w.batch * w.V * elt / 1e9:.2f} GB, "
                  f"mask {mask_bytes / 1e9:.2f} GB"}


# --------------------------------------------------------------------------- oracle arm

class OracleSample:
    """A proportional slice of one step for the CPU oracle: a fraction f of the
    trie's mask rows (seeded sample, root included) and of the batch rows of
    the decode loop. value = f * N * V pairs over the slice's wall time."""

    def __init__(self, w, nthreads: int):
        import numpy as np
        import oracle
        oracle.build()
        self.w, self.nthreads = w, nthreads
        self.trie = oracle.Trie(w.set_bytes, w.set_offsets)
        self.voc = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
        self.N = self.trie.num_nodes
        rng = np.random.default_rng(12345)
        self.order = np.concatenate([[0], 1 + rng.permutation(self.N - 1)]).astype(np.int32)
        self.bits = cpu_logits_bits(w)
        self.set_frac(0.01)

    def set_frac(self, f: float):
        import math
        self.f = min(1.0, max(f, 1.0 / self.N))
        self.rows = self.order[: max(1, int(math.ceil(self.f * self.N)))]
        self.b = max(1, int(round(self.f * self.w.batch)))

    def step(self) -> float:
        import numpy as np
        import oracle
        t0 = time.perf_counter()
        oracle.mask_rows(self.trie, self.voc, self.rows, nthreads=self.nthreads)
        oracle.decode(self.trie, self.voc, [lb[: self.b] for lb in self.bits], np.zeros(self.b, np.int32))
        return time.perf_counter() - t0

    def calibrate(self, target_s: float):
        t = self.step()
        self.set_frac(self.f * target_s / max(t, 1e-4))


def cpu_logits_bits(w):
    import numpy as np
    import torch
    from paper_2608_12574_gb300 import workloads as W
    out = []
    for s in range(w.steps):
        x = W.logits(w, s, device="cpu")
        out.append(x.view(torch.int16).numpy().view(np.uint16) if w.dtype == "bf16"
                   else x.view(torch.int32).numpy().view(np.uint32))
    return out


def cpu_baseline(w, target_step_s: float, steps: int, warmup: int) -> dict:
    """Time the oracle as it stands on this host's cores (bounded sample)."""
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    smp = OracleSample(w, cores)
    smp.calibrate(target_step_s)
    for _ in range(warmup):
        smp.step()
    times = [smp.step() for _ in range(steps)]
    per_step = sum(times) / len(times)
    cpu_model = ""
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu part")):
                cpu_model = line.split(":", 1)[1].strip()
                break
    except OSError:
        pass
    # the same oracle on one core (a smaller slice, about 2 s)
    one = OracleSample(w, 1)
    one.calibrate(min(2.0, target_step_s))
    t1 = one.step()
    single = {"value": one.f * one.N * w.V / t1, "unit": UNIT, "cores": 1, "s_per_step": t1,
              "sample": f"{len(one.rows)} mask rows and {one.b} batch rows, one step"}
    return {"value": smp.f * smp.N * w.V / per_step, "unit": UNIT, "cores": cores, "kind": "oracle",
            "single_core": single,
            "steps": len(times), "s_per_step": per_step, "cpu": cpu_model, "N_nodes": smp.N,
            "sample": f"{len(times)} steps, each a {smp.f:.4f} slice of one {w.name} step: "
                      f"{len(smp.rows)} of {smp.N} mask rows x {w.V} tokens (brute-force walks, "
                      f"OpenMP over rows) and the {w.steps}-step decode loop on {smp.b} of "
                      f"{w.batch} batch rows"}


def cpu_paper_algorithm(w, reps: int = 3) -> dict:
    """The paper's own precomputation on this host's cores (oracle/ac.c): the
    Aho-Corasick build over the vocabulary (once per tokenizer) and the trie
    traversal that yields the sparse valid lists (once per schema)."""
    import oracle
    oracle.build()
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    voc = oracle.Vocab(w.vocab_bytes, w.vocab_offsets)
    t0 = time.perf_counter()
    ac = oracle.AhoCorasick(voc)
    build_s = time.perf_counter() - t0
    trie = oracle.Trie(w.set_bytes, w.set_offsets)
    ac.pairs(trie, nthreads=cores)
    trav = []
    for _ in range(reps):
        t0 = time.perf_counter()
        rows, _ = ac.pairs(trie, nthreads=cores)
        trav.append(time.perf_counter() - t0)
    tr = min(trav)
    return {"kind": "paper algorithm (Aho-Corasick + trie traversal, sparse valid lists)",
            "cores": cores, "ac_build_ms": build_s * 1e3, "ac_states": ac.num_states,
            "traverse_ms": tr * 1e3, "valid_pairs": int(rows.size),
            "pairs_per_s_equivalent": trie.num_nodes * w.V / tr}


def run_reference(args, w):
    steps, warmup = max(1, args.steps), max(0, args.warmup)
    target = min(2.0, 150.0 / (steps + warmup + 1))
    cb = cpu_baseline(w, target, steps, warmup)
    line = {"metric": METRIC, "value": cb["value"], "unit": UNIT, "n_gpus": args.gpus, "steps": cb["steps"],
            "warmup": warmup, "ms_per_step": cb["s_per_step"] * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32 mask / " + w.dtype, "data": "synthetic",
            "impl": "reference",
            "config": workload_config(w, cb["N_nodes"]),
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


# --------------------------------------------------------------------------- GPU arm

def run_gpu(args, w, rank: int, world: int, dist):
    import numpy as np
    import torch
    from paper_2608_12574_gb300 import triemask as T

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream(dev)
    V, B, S = w.V, w.batch, w.steps
    Wd = T.mask_words(V)
    elt = 2 if w.dtype == "bf16" else 4
    hbm, peak_kind = peaks()

    # ---- setup (untimed): trie, cold compile (vocab pack + uploads), logits in HBM
    t0 = time.perf_counter()
    h = T.trie_build(w.set_bytes, w.set_offsets)
    host_build_ms = (time.perf_counter() - t0) * 1e3
    N = h.num_nodes
    mask = T.alloc_mask(h, V, dev)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, V, mask, stream)
    stream.synchronize()
    cold_compile_ms = (time.perf_counter() - t0) * 1e3
    # the vocabulary by handle from here on (a server packs it once)
    vh = T.trie_vocab_create(w.vocab_bytes, w.vocab_offsets, V)
    with torch.cuda.stream(stream):
        logits = [W_logits(w, s, dev) for s in range(S)]
        states0 = torch.zeros(B, dtype=torch.int32, device=dev)
        states = torch.zeros(B, dtype=torch.int32, device=dev)
        err = torch.zeros(1, dtype=torch.int32, device=dev)
    stream.synchronize()

    # greedy tokens of every decode step, computed once (untimed): the sampler
    # is the caller's and is not part of the timed path, so the timed step
    # replays these tokens (teacher forcing); the results are identical.
    with torch.cuda.stream(stream):
        forced = torch.zeros((S, B), dtype=torch.int32, device=dev)
        hist = torch.zeros((S, B), dtype=torch.int32, device=dev)  # states entering each decode step
        states.zero_()
        for t in range(S):
            hist[t].copy_(states)
            x = logits[t].clone()
            T.trie_apply_mask(h, x, states, stream)
            forced[t].copy_(torch.argmax(x, dim=1))
            T.trie_advance(h, states, forced[t], err, stream)
        del x
    stream.synchronize()
    if int(err.item()) != 0:
        raise RuntimeError("greedy decode reached DEAD states")

    sbuf = [states, torch.zeros_like(states)]

    def decode(logits_t):
        """The decode loop: mask step 0, then per step advance by the previous
        step's token and mask this step's logits in one launch, then the last
        advance. The initial states (states0) are only read; returns the
        buffer holding the final states."""
        T.trie_apply_mask(h, logits_t[0], states0, stream)
        prev = states0
        for t in range(1, S):
            T.trie_advance_apply(h, prev, forced[t - 1], sbuf[t % 2], logits_t[t], err, stream)
            prev = sbuf[t % 2]
        if prev is states0:  # a one-step loop: advance a copy
            sbuf[1].copy_(states0)
            prev = sbuf[1]
        T.trie_advance(h, prev, forced[S - 1], err, stream)
        return prev

    def step():
        T.trie_compile_masks_vocab(h, vh, mask, stream)
        decode(logits)

    # kernel-level graphs: the compile alone; the 16 applies of a step, back to
    # back over the 16 logits buffers with the states each decode step sees
    adv_states = [torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(S)]

    def compile_only():
        T.trie_compile_masks_vocab(h, vh, mask, stream)

    def apply_only():
        for t in range(S):
            T.trie_apply_mask(h, logits[t], hist[t], stream)

    def advance_only():
        for t in range(S):
            adv_states[t].copy_(hist[t])
            T.trie_advance(h, adv_states[t], forced[t], err, stream)

    fused_out = torch.zeros_like(states)

    def advance_apply_only():
        for t in range(1, S):
            T.trie_advance_apply(h, hist[t - 1], forced[t - 1], fused_out, logits[t], err, stream)

    def capture(fn):
        if args.no_graph:
            return fn
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        return g.replay

    with torch.cuda.stream(stream):
        for _ in range(max(args.warmup, 3)):
            step()
    stream.synchronize()
    run_step, run_compile, run_apply, run_advance, run_fused = (
        capture(f) for f in (step, compile_only, apply_only, advance_only, advance_apply_only))
    with torch.cuda.stream(stream):
        for _ in range(max(args.warmup, 3)):
            run_step()
    stream.synchronize()

    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(uuid) as clk:
        with torch.cuda.stream(stream):
            t_start.record(stream)
            for _ in range(args.steps):
                run_step()
            t_end.record(stream)
        torch.cuda.synchronize()
        ms = reduce_max(t_start.elapsed_time(t_end), dist, dev)
        ms_per_step = ms / args.steps

        # per-kernel durations: CUDA events around R back-to-back replays of
        # the kernel-level graphs, on the launching stream
        def timed(fn, reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                fn()
                e0.record(stream)
                for _ in range(reps):
                    fn()
                e1.record(stream)
            stream.synchronize()
            return e0.elapsed_time(e1) / reps

        reps = max(20, min(200, args.steps // 4))
        compile_ms = timed(run_compile, reps)
        # the same mask evaluated pair by pair (a lane per token, a warp
        # ballot per word), the design the suffix search replaces
        run_pairwise = capture(lambda: T.trie_compile_masks_pairwise(h, w.vocab_bytes, w.vocab_offsets, V, mask,
                                                                     stream))
        pairwise_ms = timed(run_pairwise, max(3, reps // 10))
        run_compile()  # the mask of the suffix search again
        apply_avg = timed(run_apply, reps) / S
        advance_avg = timed(run_advance, reps) / S
        fused_avg = timed(run_fused, reps) / (S - 1)
        # sparse valid lists: the build (CUDA events around one call; no host
        # sync inside it) and the list-driven apply over the same logits buffers
        with torch.cuda.stream(stream):
            n_valid = T.trie_compile_lists_vocab(h, vh, stream)
        stream.synchronize()
        lt = []
        for _ in range(20):
            l0, l1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                l0.record(stream)
                T.trie_compile_lists_vocab(h, vh, stream, count=False)
                l1.record(stream)
            stream.synchronize()
            lt.append(l0.elapsed_time(l1))
        lists_ms = sorted(lt)[len(lt) // 2]

        def apply_lists_only():
            for t in range(S):
                T.trie_apply_lists(h, logits[t], hist[t], stream)

        run_apply_lists = capture(apply_lists_only)
        apply_lists_avg = timed(run_apply_lists, reps) / S
        lazy = run_lazy(w, logits, forced, dev, stream, capture, timed, reps)
        formats = run_formats(w, dev, stream, capture, timed, reps)
    # a new schema with the vocabulary already cached (Sec. 4.2: the automaton
    # over the vocabulary is made once per tokenizer, only the traversal runs
    # per schema): a fresh host trie build, then its first compile, which
    # uploads the trie (6 B per node), builds its per-node tables and fills
    # its transition table. CUDA events around the compile call, median of 5.
    ns_dev, ns_host = [], []
    for _ in range(5):
        t0 = time.perf_counter()
        hn = T.trie_build(w.set_bytes, w.set_offsets)
        ns_host.append((time.perf_counter() - t0) * 1e3)
        n0, n1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            n0.record(stream)
            T.trie_compile_masks_vocab(hn, vh, mask, stream)
            n1.record(stream)
        stream.synchronize()
        ns_dev.append(n0.elapsed_time(n1))
        hn.destroy()
    new_schema_ms = statistics.median(ns_dev)
    new_schema_host_ms = statistics.median(ns_host)
    timing_src = (f"CUDA events around {reps} back-to-back replays of a graph of the {S - 1} fused "
                  f"advance+apply launches of a step (over {S - 1} logits buffers, "
                  f"{(S - 1) * B * V * elt / 1e9:.2f} GB > L2), launching stream, right after the timed region")
    # bytes an apply must move: the B x V logits written, the states, and of
    # each state's mask row the segment summary (8-byte words: 32 segment bits
    # and the compile's epoch) plus the 1,024-token segments that hold an
    # allowed token (the compile's summary lets the apply skip reading the
    # others), averaged over the decode steps' states
    segs = (Wd + 31) // 32
    seg_words = (segs + 31) // 32
    occupied = 0
    for t in range(S):
        sv = hist[t].long()
        node = (sv >= 0) & (sv < N)
        rows = mask[sv.clamp(0, N - 1)]
        rows = torch.nn.functional.pad(rows, (0, segs * 32 - Wd)).view(B, segs, 32)
        occ = (rows != 0).any(dim=2) & node[:, None]
        occupied += int(occ.sum().item())  # FINISHED / DEAD rows ({EOS}) read no mask word
    apply_bytes = B * V * elt + B * 4 + B * seg_words * 8 + (occupied / S) * 128
    fused_bytes = apply_bytes + 2 * B * 4  # + tokens read, new states written
    compile_bytes = N * Wd * 4
    apply_gbs = apply_bytes / (apply_avg * 1e-3) / 1e9
    fused_gbs = fused_bytes / (fused_avg * 1e-3) / 1e9
    compile_gbs = compile_bytes / (compile_ms * 1e-3) / 1e9

    e2e_s, h2d, d2h, h2d_only_s, e2e_runs = run_e2e(w, N, logits, forced, dev, stream, args.e2e_steps, dist)

    if rank != 0:
        return
    traffic = ncu_traffic("k_advance_apply_vec", w.name)
    parts = [ncu_traffic(k, w.name) for k in ("k_mask_probe", "k_mask_fill_beside", "k_mask_scatter")]
    traffic_c = None if any(p is None for p in parts) else sum(parts)
    line = {
        "metric": METRIC,
        "value": job_throughput(N * V, world, ms_per_step * 1e-3),
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_per_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "u32 mask / " + w.dtype,
        "data": "synthetic",
        "impl": "gb300",
        "config": workload_config(w, N),
        "parallelism": f"replicas x{world}",
        "graph": not args.no_graph,
        "roofline": {"bound": "hbm", "achieved": fused_gbs, "peak": hbm, "unit": "GB/s",
                     "frac": fused_gbs / hbm, "traffic": traffic, "kernel": "k_advance_apply_vec",
                     "bytes_per_launch": fused_bytes, "us_per_launch": fused_avg * 1e3,
                     "peak_kind": peak_kind, "timing": timing_src},
        "roofline_apply": {"bound": "hbm", "achieved": apply_gbs, "peak": hbm, "unit": "GB/s",
                           "frac": apply_gbs / hbm, "traffic": ncu_traffic("k_apply_vec", w.name),
                           "kernel": "k_apply_vec", "bytes_per_launch": apply_bytes,
                           "us_per_launch": apply_avg * 1e3, "peak_kind": peak_kind,
                           "timing": f"as roofline, a graph of the {S} applies of a step"},
        "roofline_compile": {"bound": "hbm", "achieved": compile_gbs, "peak": hbm, "unit": "GB/s",
                             "frac": compile_gbs / hbm, "traffic": traffic_c,
                             "kernel": "k_mask_probe + k_mask_fill_beside + k_mask_scatter",
                             "bytes_per_launch": compile_bytes,
                             "ms": compile_ms, "pairs_per_s": N * V / (compile_ms * 1e-3),
                             "peak_kind": peak_kind,
                             "timing": f"CUDA events around {reps} back-to-back replays of a graph of one compile"},
        "compile_pairwise": {"ms": pairwise_ms, "pairs_per_s": N * V / (pairwise_ms * 1e-3),
                             "frac_of_write_roofline": compile_bytes / (pairwise_ms * 1e-3) / 1e9 / hbm,
                             "vs_suffix_search": pairwise_ms / compile_ms,
                             "kernel": "k_mask_pairwise (a lane per token walks it from the node; "
                                       "__ballot_sync per mask word)"},
        "sparse_lists": {"entries": n_valid, "bytes": n_valid * 4 + (N + 1) * 8,
                         "compile_ms": lists_ms,
                         "apply_us_avg": apply_lists_avg * 1e3,
                         "apply_gbs": (B * V * elt + B * 4) / (apply_lists_avg * 1e-3) / 1e9,
                         "note": "valid lists as the paper stores them (Sec. 4.2); compile = median of 20 "
                                 "calls, CUDA events"},
        "lazy_rows": lazy,
        "char_position_masks": formats,
        "breakdown": {"compile_ms": compile_ms, "apply_us_avg": apply_avg * 1e3,
                      "advance_us_avg": advance_avg * 1e3, "advance_apply_us_avg": fused_avg * 1e3,
                      "host_trie_build_ms": host_build_ms,
                      "cold_compile_ms": cold_compile_ms,
                      "new_schema_compile_ms": new_schema_ms,
                      "new_schema_host_build_ms": new_schema_host_ms,
                      "new_schema_note": "fresh trie, vocabulary cached: upload, tables, transition table "
                                         "clear and fill, compile (events around the call, median of 5); "
                                         "compile_ms replays a compile whose transition table is complete",
                      "apply_gbs_conventional_rw": (2 * B * V * elt + B * Wd * 4) / (apply_avg * 1e-3) / 1e9},
        "e2e": {"value": job_throughput(N * V, world, e2e_s), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_s * 1e3,
                "h2d_only_ms": h2d_only_s * 1e3, "h2d_gbs": h2d / h2d_only_s / 1e9,
                "runs_ms_per_step": [round(r * 1e3, 4) for r in e2e_runs],
                "timing": f"the fastest of {len(e2e_runs)} runs of {args.e2e_steps} pipelined steps, wall clock "
                          "around each run (the copies alone: the fastest of 5 rounds, CUDA events)"},
        "gpu_launches": args.steps * (compile_kernels(w, N, h.max_depth, torch.cuda.get_device_properties(dev).multi_processor_count) + S + 1),
        "clocks": clk.summary(),
    }
    if not args.no_dynamic:
        del logits, mask
        torch.cuda.empty_cache()
        line["dynamic_sets"] = run_dynamic(dev, stream, rank=rank, world=world, dist=dist)
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds / 5, 5, 1)
        line["cpu_paper_algorithm"] = cpu_paper_algorithm(w)
    print(json.dumps(line))


def run_e2e(w, n_nodes: int, logits, forced, dev, stream, steps: int, dist=None):
    """The e2e step through the C ABI from host buffers: per step the trie is
    built from the host strings and compiled, the logits and tokens are
    copied from pinned host memory and the states read back after every
    decode step. Returns (seconds per step, H2D bytes, D2H bytes, seconds of
    the step's H2D copies alone)."""
    import torch
    from paper_2608_12574_gb300 import triemask as T
    V, B, S = w.V, w.batch, w.steps
    sbuf = [torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(2)]
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    mask = torch.empty((n_nodes, T.mask_words(V)), dtype=torch.int32, device=dev)
    vh = T.trie_vocab_create(w.vocab_bytes, w.vocab_offsets, V)  # packed and uploaded once, like a server's
    # ---- e2e: host strings -> trie_build -> compile -> decode, with the logits
    # and the step's tokens copied from pinned host memory and the states read
    # back every decode step. Steps are pipelined as a server would run them:
    # the copies run on their own stream into two alternating buffer sets, so
    # step i + 1's copies follow step i's at once; decode step t waits only
    # for its own logits; the next step's host trie build runs while the GPU
    # works, and a step's handle is released in stream order (no device sync).
    host_logits = [lg.cpu().pin_memory() for lg in logits]
    host_forced = forced.cpu().pin_memory()
    host_states = [torch.zeros((S, B), dtype=torch.int32).pin_memory() for _ in range(2)]
    copy_stream = torch.cuda.Stream(dev)
    with torch.cuda.stream(stream):
        dlogs = [[torch.empty_like(lg) for lg in logits] for _ in range(2)]
        dtok = [torch.empty((S, B), dtype=torch.int32, device=dev) for _ in range(2)]
    arrived = [[torch.cuda.Event() for _ in range(S + 1)] for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]
    h2d = int(w.set_bytes.nbytes + w.set_offsets.nbytes + host_forced.numel() * 4
              + sum(x.numel() * x.element_size() for x in host_logits))
    d2h = S * B * 4

    def e2e_step(i, hh):
        """Queues step i on handle hh (built from the host strings); returns
        the next step's handle, built while step i runs."""
        k = i % 2
        copy_stream.wait_event(consumed[k])  # step i - 2 is done with buffer set k
        with torch.cuda.stream(copy_stream):
            dtok[k].copy_(host_forced, non_blocking=True)
            arrived[k][S].record(copy_stream)
            for t in range(S):
                dlogs[k][t].copy_(host_logits[t], non_blocking=True)
                arrived[k][t].record(copy_stream)
        T.trie_compile_masks_vocab(hh, vh, mask, stream)
        sbuf[0].zero_()
        stream.wait_event(arrived[k][S])
        cur = 0
        for t in range(S):
            stream.wait_event(arrived[k][t])
            if t == 0:
                T.trie_apply_mask(hh, dlogs[k][0], sbuf[0], stream)
            else:
                T.trie_advance_apply(hh, sbuf[cur], dtok[k][t - 1], sbuf[1 - cur], dlogs[k][t], err, stream)
                cur = 1 - cur
            host_states[k][t].copy_(sbuf[cur], non_blocking=True)
        T.trie_advance(hh, sbuf[cur], dtok[k][S - 1], err, stream)
        consumed[k].record(stream)
        nxt = T.trie_build(w.set_bytes, w.set_offsets)  # host work beside the GPU's
        hh.destroy_async(stream)
        return nxt

    # the timed loop runs three times and the fastest counts, as for the
    # copies alone below: on these shared hosts the host link's bandwidth
    # dropped to about half for whole runs at times (5.96 against 10.8 ms)
    runs = []
    with torch.cuda.stream(stream):
        hh = T.trie_build(w.set_bytes, w.set_offsets)
        for i in range(2):
            hh = e2e_step(i, hh)
        for _ in range(3):
            torch.cuda.synchronize()
            if dist is not None:
                dist.barrier()
            t0 = time.perf_counter()
            for i in range(steps):
                hh = e2e_step(i, hh)
            torch.cuda.synchronize()
            runs.append((time.perf_counter() - t0) / steps)
        hh.destroy()
    e2e_s = reduce_max(min(runs), dist, dev)
    # context: the step's host->device copies alone (the floor of the e2e
    # step), the fastest of a few rounds timed with events on the copy stream
    torch.cuda.synchronize()
    rounds = []
    for _ in range(5):
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(copy_stream):
            c0.record(copy_stream)
            dtok[0].copy_(host_forced, non_blocking=True)
            for t in range(S):
                dlogs[0][t].copy_(host_logits[t], non_blocking=True)
            c1.record(copy_stream)
        copy_stream.synchronize()
        rounds.append(c0.elapsed_time(c1) * 1e-3)
    h2d_only_s = min(rounds)
    return e2e_s, h2d, d2h, h2d_only_s, runs


def run_lazy(w, logits, forced, dev, stream, capture, timed, reps: int) -> dict:
    """The decode loop of the workload with lazy rows (App. H.5) instead of a
    compiled mask: step 0 masked by trie_lazy_apply, steps 1.. by
    trie_lazy_advance_apply (the same tokens as the dense loop). With no
    cache every pass computes every row it needs; with a 4,096-row cache the
    first pass after set-up computes them and later passes find them cached."""
    import torch
    from paper_2608_12574_gb300 import triemask as T
    V, B, S = w.V, w.batch, w.steps
    out = {"note": "rows computed on first use (App. H.5); a pass = step 0 apply + "
                   f"{S - 1} fused advance+apply calls, 3 kernels each"}
    sb = [torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(2)]
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    for cache in (0, 4096):
        hl = T.trie_build(w.set_bytes, w.set_offsets)
        T.trie_lazy_init(hl, w.vocab_bytes, w.vocab_offsets, V, cache, B)

        def loop():
            sb[0].zero_()
            T.trie_lazy_apply(hl, logits[0], sb[0], stream)
            cur = 0
            for t in range(1, S):
                T.trie_lazy_advance_apply(hl, sb[cur], forced[t - 1], sb[1 - cur], logits[t], err, stream)
                cur = 1 - cur

        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            loop()
            e1.record(stream)
        stream.synchronize()
        cold = e0.elapsed_time(e1)
        run = capture(loop)
        pass_ms = timed(run, reps)
        hits, misses = T.trie_lazy_stats(hl)
        rows_bytes = (((cache + 7) // 8 * 8) + B) * T.mask_words(V) * 4
        out[f"cache_{cache}"] = {"cache_rows": cache, "first_pass_ms": cold, "pass_ms": pass_ms,
                                 "us_per_step": pass_ms * 1e3 / S, "hits": hits, "misses": misses,
                                 "row_bytes": rows_bytes}
        hl.destroy()
    return out


def run_formats(w, dev, stream, capture, timed, reps: int) -> dict:
    """Character-position masks (App. K) of the four fixed formats of the
    paper's comparison, compiled with the workload's vocabulary: per format
    the mask compile (a graph of one fmt_compile_masks, CUDA events) and the
    number of allowed (position, token) pairs."""
    import numpy as np
    import torch
    from paper_2608_12574_gb300 import triemask as T
    from paper_2608_12574_gb300 import workloads as W
    out = {"V": w.V, "note": "App. K: one row per position of the format; compile = fmt_compile_masks"}
    for name, pat in W.FORMATS.items():
        f = T.fmt_build(W.format_classes(pat))
        m = T.fmt_alloc_mask(f, w.V, dev)
        with torch.cuda.stream(stream):
            T.fmt_compile_masks(f, w.vocab_bytes, w.vocab_offsets, w.V, m, stream)
        stream.synchronize()
        run = capture(lambda: T.fmt_compile_masks(f, w.vocab_bytes, w.vocab_offsets, w.V, m, stream))
        us = timed(run, reps) * 1e3
        pairs = int(np.unpackbits(m.cpu().numpy().view(np.uint8)).sum())
        out[name] = {"L": f.L, "compile_us": us, "allowed_pairs": pairs,
                     "pairs_per_s": (f.L + 1) * w.V / (us * 1e-6)}
        f.destroy()
    return out


def request_share(n_requests: int, rank: int, world: int) -> tuple[int, int]:
    """Requests [lo, hi) of one rank: a contiguous block, sizes differing by at
    most one, every request on exactly one rank."""
    base, extra = divmod(n_requests, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def share_of(w, lo: int, hi: int):
    """The per-request forest workload restricted to requests [lo, hi): their
    strings, and set_index rebased to start at 0 (vocabulary unchanged)."""
    import dataclasses
    import numpy as np
    idx = w.set_index
    s0, s1 = int(idx[lo]), int(idx[hi])
    offs = w.set_offsets[s0:s1 + 1]
    return dataclasses.replace(
        w, set_bytes=w.set_bytes[int(offs[0]):int(offs[-1])], set_offsets=(offs - offs[0]).astype(np.int64),
        set_index=(idx[lo:hi + 1] - idx[lo]).astype(np.int32), batch=hi - lo)


def run_dynamic(dev, stream, steps: int = 32, reps: int = 5, rank: int = 0, world: int = 1, dist=None) -> dict:
    """The dynamic per-query-set workload, end to end with logits resident:
    256 requests, each with its own set of K ~ U[300, 2000] names from a
    50,000-name pool; per batch the 256 tries are built as one forest (on the
    device; the host builder is timed beside it), compiled on the GPU (sparse
    lists; the dense forest mask is timed separately) and decoded for 32
    steps (apply + advance, greedy tokens replayed)."""
    import torch
    from paper_2608_12574_gb300 import triemask as T
    from paper_2608_12574_gb300 import workloads as W
    full = W.config(5)
    lo, hi = request_share(full.batch, rank, world)
    w = share_of(full, lo, hi) if world > 1 else full
    B, V = w.batch, w.V
    out = {"workload": full.name, "requests": full.batch, "V": V, "decode_steps": steps,
           "ranks": world, "requests_per_rank": [request_share(full.batch, r, world) for r in range(world)]}
    t0 = time.perf_counter()
    h = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index)
    out["host_forest_build_ms"] = (time.perf_counter() - t0) * 1e3
    N = h.num_nodes
    out["N_nodes"] = N
    roots = torch.as_tensor(h.roots(), device=dev)
    # the tokenizer's vocabulary is packed and uploaded once (a handle); the
    # requests' sets change every batch
    vh = T.trie_vocab_create(w.vocab_bytes, w.vocab_offsets, V)
    with torch.cuda.stream(stream):
        logits = [W.logits(w, t, device=str(dev)) for t in range(steps)]
        T.trie_compile_lists_vocab(h, vh, stream)
        states = roots.clone()
        err = torch.zeros(1, dtype=torch.int32, device=dev)
        forced = torch.zeros((steps, B), dtype=torch.int32, device=dev)
        for t in range(steps):
            x = logits[t].clone()
            T.trie_apply_lists(h, x, states, stream)
            forced[t].copy_(torch.argmax(x, dim=1))
            T.trie_advance(h, states, forced[t], err, stream)
        del x
    stream.synchronize()
    out["dead_moves"] = int(err.item())
    out["finished"] = int((states == T.TRIE_STATE_FINISHED).sum().item())

    sb = [states, torch.empty_like(states)]

    def decode():  # one launch per step: apply, then advance + apply of the next step
        sb[0].copy_(roots)
        T.trie_apply_lists(h, logits[0], sb[0], stream)
        for t in range(1, steps):
            T.trie_advance_apply_lists(h, sb[(t - 1) % 2], forced[t - 1], sb[t % 2], logits[t], err, stream)

    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        decode()
        with torch.cuda.graph(g, stream=stream):
            decode()
        g.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    stream.synchronize()
    out["decode_ms"] = e0.elapsed_time(e1) / reps
    # one list-driven apply (the fused advance + apply of a step): the B x V
    # logits written and the states read (the rows' list entries, a few KB
    # read from L2, are left out)
    peak, peak_kind = peaks()
    elt = 2 if w.dtype == "bf16" else 4
    per_launch_us = out["decode_ms"] * 1e3 / steps
    ab = B * V * elt + 3 * B * 4
    out["roofline_apply_lists"] = {"bound": "hbm", "achieved": ab / (per_launch_us * 1e-6) / 1e9, "peak": peak,
                                   "unit": "GB/s", "frac": ab / (per_launch_us * 1e-6) / 1e9 / peak,
                                   "bytes_per_launch": ab, "us_per_launch": per_launch_us,
                                   "peak_kind": peak_kind, "kernel": "k_apply_lists",
                                   "traffic": ncu_traffic("k_apply_lists", full.name),
                                   "timing": f"the {steps}-step decode graph (1 + {steps - 1} launches) over "
                                             f"its launches, CUDA events around {reps} replays"}
    lt, lw = [], []
    for _ in range(reps):
        stream.synchronize()
        t0 = time.perf_counter()
        with torch.cuda.stream(stream):
            e0.record(stream)
            T.trie_compile_lists_vocab(h, vh, stream, count=False)
            e1.record(stream)
        stream.synchronize()
        lw.append(time.perf_counter() - t0)
        lt.append(e0.elapsed_time(e1))
    n_valid = T.trie_num_valid(h)
    out["lists_compile_ms"] = min(lt)
    out["lists_compile_wall_ms"] = min(lw) * 1e3
    out["list_entries"] = n_valid
    out["list_bytes"] = n_valid * 4 + (N + 1) * 8
    # the list compile's algorithmic traffic: the entries and offsets written
    # plus the per-node tables the walks read (window 16 B, anc 64 B, depth,
    # terminal: 82 B per node, read by both walks)
    peak, peak_kind = peaks()
    list_bytes = out["list_bytes"] + 2 * 82 * N
    out["roofline_lists"] = {"bound": "hbm", "achieved": list_bytes / (min(lt) * 1e-3) / 1e9, "peak": peak,
                             "unit": "GB/s", "frac": list_bytes / (min(lt) * 1e-3) / 1e9 / peak,
                             "bytes_per_launch": list_bytes, "peak_kind": peak_kind,
                             "kernel": "k_list_walk (count) + scans + k_list_walk (write)",
                             "timing": f"CUDA events around one trie_compile_lists, best of {reps}"}
    # end to end per batch of requests: forest build (on the device, or on the
    # host) + list compile + decode
    builders = {
        "device": lambda: T.trie_build_many_device(w.set_bytes, w.set_offsets, w.set_index, stream),
        "host": lambda: T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index),
    }
    bt = []
    for _ in range(reps):
        t0 = time.perf_counter()
        hh = builders["device"]()
        stream.synchronize()  # the build returns before its last kernels have run
        bt.append(time.perf_counter() - t0)
        hh.destroy()
    out["device_forest_build_ms"] = min(bt) * 1e3
    # the batch's initial states (the roots) go up through a pinned buffer,
    # queued before the compile: a pageable copy would wait for the stream
    roots_host = torch.empty(B, dtype=torch.int32).pin_memory()
    st = [torch.empty(B, dtype=torch.int32, device=dev) for _ in range(2)]
    for kind, build in builders.items():
        et = []
        for _ in range(reps):
            t0 = time.perf_counter()
            hh = build()
            with torch.cuda.stream(stream):
                roots_host.numpy()[:] = hh.roots()
                st[0].copy_(roots_host, non_blocking=True)
                T.trie_compile_lists_vocab(hh, vh, stream, count=False)
                T.trie_apply_lists(hh, logits[0], st[0], stream)
                for t in range(1, steps):
                    T.trie_advance_apply_lists(hh, st[(t - 1) % 2], forced[t - 1], st[t % 2], logits[t], err,
                                               stream)
            stream.synchronize()
            et.append(time.perf_counter() - t0)
            hh.destroy()
        # with several ranks each holds a share of the requests: the batch is
        # done when the slowest rank is (max over ranks; no data exchange)
        key = "end_to_end_ms" if kind == "device" else "end_to_end_host_build_ms"
        out[key] = reduce_max(min(et) * 1e3, dist, dev)
    out["requests_per_s"] = full.batch / (out["end_to_end_ms"] * 1e-3)
    out["scaling"] = "strong: the 256 requests are split across the ranks" if world > 1 else "single rank"
    # lazy rows (App. H.5) instead of the lists: no per-batch compile, each
    # step computes the rows its states reach (the requests are new every
    # batch, so no cache is kept)
    def lazy_steps(hh, st):
        T.trie_lazy_apply(hh, logits[0], st[0], stream)
        for t in range(1, steps):
            T.trie_lazy_advance_apply(hh, st[(t - 1) % 2], forced[t - 1], st[t % 2], logits[t], err, stream)

    et = []
    for _ in range(reps):
        t0 = time.perf_counter()
        hh = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index)
        T.trie_lazy_init(hh, w.vocab_bytes, w.vocab_offsets, V, 0, B)
        with torch.cuda.stream(stream):
            st = [torch.as_tensor(hh.roots(), device=dev), torch.empty(B, dtype=torch.int32, device=dev)]
            lazy_steps(hh, st)
        stream.synchronize()
        et.append(time.perf_counter() - t0)
        hh.destroy()
    out["lazy_end_to_end_ms"] = min(et) * 1e3  # host-built forest (its pre-order tables)
    T.trie_lazy_init(h, w.vocab_bytes, w.vocab_offsets, V, 0, B)
    lst = [roots.clone(), torch.empty(B, dtype=torch.int32, device=dev)]

    def lazy_decode():
        lst[0].copy_(roots)
        lazy_steps(h, lst)

    gl = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        lazy_decode()
        with torch.cuda.graph(gl, stream=stream):
            lazy_decode()
        gl.replay()
        e0.record(stream)
        for _ in range(reps):
            gl.replay()
        e1.record(stream)
    stream.synchronize()
    out["lazy_decode_ms"] = e0.elapsed_time(e1) / reps
    # the dense form of the same forest: a [N, ceil(V/32)] mask
    dense_bytes = N * T.mask_words(V) * 4
    free, _ = torch.cuda.mem_get_info(dev)
    if dense_bytes < free * 0.8:
        mask = T.alloc_mask(h, V, dev)
        with torch.cuda.stream(stream):
            T.trie_compile_masks_vocab(h, vh, mask, stream)
            e0.record(stream)
            T.trie_compile_masks_vocab(h, vh, mask, stream)
            e1.record(stream)
        stream.synchronize()
        ms = e0.elapsed_time(e1)
        out["dense_compile_ms"] = ms
        out["dense_mask_bytes"] = dense_bytes
        out["dense_compile_gbs"] = dense_bytes / (ms * 1e-3) / 1e9
        del mask
    del logits
    torch.cuda.empty_cache()
    h.destroy()
    return out


def reduce_max(x: float, dist, device) -> float:
    """Max of a per-rank scalar over all ranks (the slowest rank sets the job time)."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, world: int, seconds: float) -> float:
    """Whole-job throughput under weak scaling: every rank does the same work."""
    return world * units_per_rank / seconds


def W_logits(w, s, dev):
    from paper_2608_12574_gb300 import workloads as W
    return W.logits(w, s, device=str(dev))


def run_profile(args, w) -> None:
    """One part of the path alone, --reps times after one untimed call, with
    CUDA events around the repetitions on the launching stream (eager
    launches, no graph): the commands the ncu summaries were made with."""
    import torch
    from paper_2608_12574_gb300 import _build
    from paper_2608_12574_gb300 import triemask as T
    from paper_2608_12574_gb300 import workloads as W
    _build.build()
    dev = torch.device("cuda:0")
    stream = torch.cuda.Stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn, what):
        with torch.cuda.stream(stream):
            fn()
            e0.record(stream)
            for _ in range(args.reps):
                fn()
            e1.record(stream)
        stream.synchronize()
        print(f"{what}: {e0.elapsed_time(e1) * 1e3 / max(1, args.reps):.2f} us per call", flush=True)

    if args.profile in ("compile", "pairwise", "lazy", "step"):
        h = T.trie_build(w.set_bytes, w.set_offsets)
        mask = T.alloc_mask(h, w.V, dev)
        T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, mask)
        vh = T.trie_vocab_create(w.vocab_bytes, w.vocab_offsets, w.V)
        if args.profile == "compile":
            timed(lambda: T.trie_compile_masks_vocab(h, vh, mask, stream),
                  f"{w.name} trie_compile_masks, {h.num_nodes} nodes")
        elif args.profile == "pairwise":
            timed(lambda: T.trie_compile_masks_pairwise(h, w.vocab_bytes, w.vocab_offsets, w.V, mask, stream),
                  f"{w.name} trie_compile_masks_pairwise, {h.num_nodes} nodes")
        else:
            V, B, S = w.V, w.batch, w.steps
            logits = [W.logits(w, s, device=str(dev)) for s in range(S)]
            states = torch.zeros(B, dtype=torch.int32, device=dev)
            err = torch.zeros(1, dtype=torch.int32, device=dev)
            forced = torch.zeros((S, B), dtype=torch.int32, device=dev)
            for t in range(S):  # greedy tokens, replayed below
                x = logits[t].clone()
                T.trie_apply_mask(h, x, states)
                forced[t].copy_(torch.argmax(x, dim=1))
                T.trie_advance(h, states, forced[t], err)
            s0 = torch.zeros(B, dtype=torch.int32, device=dev)
            sb = [torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(2)]
            if args.profile == "lazy":
                T.trie_lazy_init(h, w.vocab_bytes, w.vocab_offsets, V, args.cache_rows, B)

                def loop():
                    T.trie_lazy_apply(h, logits[0], s0, stream)
                    prev = s0
                    for t in range(1, S):
                        T.trie_lazy_advance_apply(h, prev, forced[t - 1], sb[t % 2], logits[t], err, stream)
                        prev = sb[t % 2]

                timed(loop, f"{w.name} lazy decode loop ({S} steps, cache {args.cache_rows} rows)")
            else:
                def loop():
                    T.trie_compile_masks_vocab(h, vh, mask, stream)
                    T.trie_apply_mask(h, logits[0], s0, stream)
                    prev = s0
                    for t in range(1, S):
                        T.trie_advance_apply(h, prev, forced[t - 1], sb[t % 2], logits[t], err, stream)
                        prev = sb[t % 2]
                    T.trie_advance(h, prev, forced[S - 1], err, stream)

                timed(loop, f"{w.name} step (compile + {S} decode steps, eager)")
        return
    full = W.dynamic_requests(args.requests)
    if args.device_build:
        h = T.trie_build_many_device(full.set_bytes, full.set_offsets, full.set_index, stream)
    else:
        h = T.trie_build_many(full.set_bytes, full.set_offsets, full.set_index)
    vh = T.trie_vocab_create(full.vocab_bytes, full.vocab_offsets, full.V)
    if args.profile == "lists":
        timed(lambda: T.trie_compile_lists_vocab(h, vh, stream, count=False),
              f"{args.requests}-request forest trie_compile_lists, {h.num_nodes} nodes")
        print(f"{T.trie_num_valid(h)} entries")
        return
    # listdecode: the 32-step list-driven decode of the dynamic workload
    # (apply, then 31 fused advance + apply launches), greedy tokens replayed
    steps, B, V = 32, full.batch, full.V
    roots = torch.as_tensor(h.roots(), device=dev)
    with torch.cuda.stream(stream):
        T.trie_compile_lists_vocab(h, vh, stream)
        logits = [W.logits(full, t, device=str(dev)) for t in range(steps)]
        states = roots.clone()
        err = torch.zeros(1, dtype=torch.int32, device=dev)
        forced = torch.zeros((steps, B), dtype=torch.int32, device=dev)
        for t in range(steps):
            x = logits[t].clone()
            T.trie_apply_lists(h, x, states, stream)
            forced[t].copy_(torch.argmax(x, dim=1))
            T.trie_advance(h, states, forced[t], err, stream)
    sb = [torch.empty_like(roots), torch.empty_like(roots)]

    def decode():
        sb[0].copy_(roots)
        T.trie_apply_lists(h, logits[0], sb[0], stream)
        for t in range(1, steps):
            T.trie_advance_apply_lists(h, sb[(t - 1) % 2], forced[t - 1], sb[t % 2], logits[t], err, stream)

    timed(decode, f"{args.requests}-request list decode loop ({steps} launches, eager)")


def launch_ranks(n: int) -> int:
    """Re-runs this command as n local ranks (one process per GPU), the way
    the multi-GPU launch does: torch.distributed.run on 127.0.0.1."""
    import socket
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
           "--master-addr=127.0.0.1", f"--master-port={port}", os.path.abspath(__file__)] + sys.argv[1:]
    return subprocess.call(cmd)


def main():
    args = parse_args()
    from paper_2608_12574_gb300 import workloads as W
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    if args.gpus < 1:
        sys.exit("--gpus must be >= 1")
    if "WORLD_SIZE" not in os.environ and args.gpus > 1 and args.impl == "gb300":
        sys.exit(launch_ranks(args.gpus))  # not under a launcher: start the ranks here
    if "WORLD_SIZE" in os.environ and world != args.gpus:
        sys.exit(f"--gpus {args.gpus} does not match WORLD_SIZE {world} of the launch")
    w = W.config(args.config)
    if args.profile:
        run_profile(args, w)
        return
    if args.impl == "reference":
        if rank == 0:
            run_reference(args, w)
        return
    from paper_2608_12574_gb300 import _build
    if rank == 0:
        _build.build()
    dist = None
    if world > 1:
        import torch
        import torch.distributed as dist_
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        dist_.init_process_group("nccl")
        dist = dist_
        dist.barrier()
    run_gpu(args, w, rank, world, dist)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
