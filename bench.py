"""Benchmark of the verify step on GB300: prints ONE JSON line.

Workload: the 8B-class target verify step of the paper's speculative-decoding
loop (Sec. 3.2 Eq. verify; target shape from Sec. 5 "Targets and drafts":
Qwen3-VL-8B backbone, 36 layers). Per scene and step, every one of the 36
layers runs, on its own KV cache (L = 4096 prefix = 4 cameras x 896 patches +
512 text tokens, 32 query / 8 KV heads x 128, bf16):
    M-RoPE of the K + 1 = 8 new Q/K rows (sections [16,24,24], base 1e6)
    KV append of the 8 rows
    verify attention of the 8 causal rows over 4104 keys
then one greedy acceptance over bf16 logits [8, 151936] and the KV rollback
of all 36 layers to the committed length. After the timed work of a step the
lengths are put back to L (one 144-byte device copy) so that every step
processes the same L = 4096 workload.

Each layer is one sd_verify_layer call (M-RoPE + append + attention in one
tcgen05 kernel); layers after the first are programmatic dependent launches
that stream their cached prefix while the previous layer still runs.
The 36 caches (605 MB) exceed the 129 MB L2, so every step streams its KV
from HBM: "inputs larger than L2". The whole step is captured once in a CUDA
graph and replayed. Multi-GPU: one independent replica per rank (scenes are
independent: weak scaling, no data-path collective).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
    python bench.py --sweep     # sd_verify_attention over the batched sweep grid
    python bench.py --floor     # launch and streaming floors of the chained layers
"""

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verify-step µs & HBM GB/s vs ~8 TB/s at L=4096,K=7,32q/8kv; accept µs"
LAYERS = 36
L, K, HQ, HKV, D, V = 4096, 7, 32, 8, 128, 151936
R = K + 1
SECTIONS = (16, 24, 24)
BASE = 1e6


# ------------------------------------------------------------ byte accounting
def attention_bytes(B=1):
    """Algorithmic bytes of one verify-attention launch: K and V of L + R keys
    for every KV head, plus the Q rows read and the O rows written."""
    kv = B * (L + R) * HKV * D * 2 * 2
    qo = 2 * B * R * HQ * D * 2
    return kv + qo


def layer_bytes(B=1):
    rope = 2 * B * R * (HQ + HKV) * D * 2          # read + write Q and K rows
    append = 2 * 2 * B * R * HKV * D * 2           # read K/V rows, write them
    return attention_bytes(B) + rope + append


def step_bytes(B=1):
    accept = B * R * V * 2 + B * K * 4 + B * (2 * R + 1) * 4
    rollback = 2 * LAYERS * B * 4 + B * 4
    return LAYERS * layer_bytes(B) + accept + rollback


# ------------------------------------------------------------------ helpers
def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def kernel_source_hash():
    path = os.path.join(ROOT, "paper_2606_31160_gb300", "csrc", "attention_tc.cu")
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def ncu_traffic(kernel="verify_layer"):
    """DRAM bytes per launch of the given kernel from the committed ncu
    summary, or None when the kernel source changed since the counters were
    taken."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)[kernel]
        if d.get("src_sha256") == kernel_source_hash():
            return float(d["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    FIELDS = ["clocks.sm", "clocks.max.sm", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap"]
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, index):
        self.index = index
        self.samples = []
        self._stop = threading.Event()
        self._thread = None

    def _one(self):
        try:
            out = subprocess.run(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + ",".join(self.FIELDS),
                                  "--format=csv,noheader,nounits"], capture_output=True, text=True, timeout=5)
            parts = [p.strip() for p in out.stdout.strip().split(",")]
            if len(parts) == len(self.FIELDS):
                self.samples.append(parts)
        except Exception:
            pass

    def _run(self):
        while not self._stop.is_set():
            self._one()
            self._stop.wait(0.1)

    def __enter__(self):
        self._thread = threading.Thread(target=self._run, daemon=True)
        self._thread.start()
        return self

    def __exit__(self, *exc):
        self._stop.set()
        self._thread.join(timeout=10)
        if not self.samples:
            self._one()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        sm = [float(s[0]) for s in self.samples if s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in self.samples if s[1].replace(".", "").isdigit()]
        reasons = set()
        for s in self.samples:
            for name, val in zip(self.NAMES, s[2:]):
                if val.strip().lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(self.samples)}


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


# ------------------------------------------------------------- ranks
# The verify step shards by scene: every rank runs whole scenes of its own
# (weak scaling, no data-path collective). These helpers are the only
# multi-rank logic; tests/test_dist_gloo.py runs them on two gloo ranks.
def scenes_of_rank(scenes_per_rank, rank):
    """Global scene indices a rank verifies: a contiguous block of its own."""
    return list(range(rank * scenes_per_rank, (rank + 1) * scenes_per_rank))


def max_over_ranks(value, world, device="cpu"):
    """The slowest rank's time (the job's time): all-reduce MAX."""
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_gbs(bytes_per_rank, world, ms_per_step):
    """Whole-job throughput: the bytes every rank verified / the slowest rank's time."""
    return bytes_per_rank * world / (ms_per_step * 1e-3) / 1e9


# ------------------------------------------------------------- workload
class Step:
    """Device-resident inputs and outputs of one verify step (one scene)."""

    def __init__(self, device, scene=0):
        from paper_2606_31160_gb300 import sd, workloads
        self.sd = sd
        self.device = device
        gen_t0 = time.time()
        self.cases = [workloads.target_layer(B=1, layer=l, ell=[3], scene=scene) for l in range(LAYERS)]
        self.gen_s = time.time() - gen_t0
        c0 = self.cases[0]
        # the per-step inputs live in one device buffer, and their host copies
        # (the end-to-end leg's source) in one pinned buffer of the same layout,
        # so that a step's inputs travel in a single copy
        parts = [("q", torch.stack([c.q for c in self.cases])),         # [36,1,R,HQ,D]
                 ("k", torch.stack([c.k_new for c in self.cases])),
                 ("v", torch.stack([c.v_new for c in self.cases])),
                 ("pos", c0.pos), ("logits", c0.extra["logits"]), ("draft", c0.extra["draft"])]
        offs, off = [], 0
        for _, t in parts:
            offs.append(off)
            off += (t.numel() * t.element_size() + 255) // 256 * 256
        self.h_in = torch.empty(off, dtype=torch.uint8).pin_memory()
        self.d_in = torch.empty(off, dtype=torch.uint8, device=device)
        for (name, t), o in zip(parts, offs):
            n = t.numel() * t.element_size()
            h = self.h_in[o:o + n].view(t.dtype).view(t.shape)
            h.copy_(t)
            setattr(self, name, self.d_in[o:o + n].view(t.dtype).view(t.shape))
        self.d_in.copy_(self.h_in)
        self.lens = torch.full((LAYERS, 1), L, dtype=torch.int32, device=device)
        self.lens0 = self.lens.clone()
        self.caches = [sd.KVCache(c.k_cache.to(device), c.v_cache.to(device), self.lens[l])
                       for l, c in enumerate(self.cases)]
        self.out = torch.empty_like(self.q)
        self.ws = sd.workspace(sd.greedy_workspace_bytes(1, K, V), device)
        need = sd.layer_workspace_bytes(1, R, HQ, HKV, D, self.caches[0].shape[2])
        self.ws_layer = [sd.workspace(need, device) for _ in range(LAYERS)]
        # the step's result (n_emit, then the R tokens) in one buffer: one copy back
        self.res = torch.zeros((1 + R,), dtype=torch.int32, device=device)
        self.n_emit = self.res[:1]
        self.tokens = self.res[1:].view(1, R)
        self.argmax = torch.zeros((1, R), dtype=torch.int32, device=device)
        self.h_out = torch.zeros((1 + R,), dtype=torch.int32).pin_memory()
        for c in self.cases:  # free host copies of the caches
            c.k_cache = c.v_cache = None

    def layers(self):
        for l in range(LAYERS):
            self.sd.verify_layer(self.q[l], self.k[l], self.v[l], self.pos, SECTIONS, self.caches[l], 0, BASE,
                                 out=self.out[l], ws=self.ws_layer[l], early=l > 0)

    def run(self):
        sd = self.sd
        self.layers()
        sd.accept_greedy(self.logits, self.draft, ws=self.ws, n_emit=self.n_emit, tokens=self.tokens,
                         argmax=self.argmax)
        sd.kv_rollback(self.lens, self.n_emit, R)
        self.lens.copy_(self.lens0, non_blocking=True)

    def run_unfused(self):
        """The same step with rope, append and attention as separate kernels."""
        sd = self.sd
        for l in range(LAYERS):
            sd.rope_apply(self.q[l], self.k[l], self.pos, SECTIONS, 0, BASE)
            sd.kv_append(self.caches[l], self.k[l], self.v[l])
            sd.verify_attention(self.q[l], self.caches[l], out=self.out[l])
        sd.accept_greedy(self.logits, self.draft, ws=self.ws, n_emit=self.n_emit, tokens=self.tokens,
                         argmax=self.argmax)
        sd.kv_rollback(self.lens, self.n_emit, R)
        self.lens.copy_(self.lens0, non_blocking=True)

    def layers_only(self):
        """The 36 fused layer launches alone, lengths put back after them."""
        self.layers()
        self.lens.copy_(self.lens0, non_blocking=True)

    def attention_only(self, early=True):
        """The standalone sd_verify_attention over the 36 appended caches; layers
        after the first are programmatic dependent launches (SD_ATTN_PREFIX_EARLY)
        unless early=False."""
        for l in range(LAYERS):
            self.sd.verify_attention(self.q[l], self.caches[l], out=self.out[l], early=early and l > 0)

    def accept_only(self):
        self.sd.accept_greedy(self.logits, self.draft, ws=self.ws, n_emit=self.n_emit, tokens=self.tokens,
                              argmax=self.argmax)

    ACCEPT_COPIES = 64  # 64 x 2.43 MB of logits > L2

    def accept_chain(self):
        """ACCEPT_COPIES greedy accepts back to back, each over its own copy of
        the logits (allocated on first use)."""
        if not hasattr(self, "logit_copies"):
            self.logit_copies = [self.logits.clone() for _ in range(self.ACCEPT_COPIES)]
        for lg in self.logit_copies:
            self.sd.accept_greedy(lg, self.draft, ws=self.ws, n_emit=self.n_emit, tokens=self.tokens,
                                  argmax=self.argmax)

    def h2d(self):
        self.d_in.copy_(self.h_in, non_blocking=True)

    def d2h(self):
        self.h_out.copy_(self.res, non_blocking=True)

    @property
    def h2d_bytes(self):
        return self.h_in.numel()  # the inputs and the 256-byte alignment between them

    @property
    def d2h_bytes(self):
        return self.h_out.numel() * 4


def capture(fn):
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn()  # warm once on the capture stream
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    with torch.cuda.graph(g):
        fn()
    torch.cuda.synchronize()
    return g


def time_graph(g, reps, warm=3):
    for _ in range(warm):
        g.replay()
    torch.cuda.synchronize()
    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(reps):
        g.replay()
    e1.record(st)
    e1.synchronize()
    return e0.elapsed_time(e1) / reps  # ms


# ------------------------------------------------------------- CPU oracle
def time_sample_accept(device, reps=20):
    """sd_accept_sample on the stochastic-acceptance workload (B=8, K=7,
    V=151936, T=0.6, fp32 target and draft logits: 72.9 MB a call): graph of
    calls alternating over two copies of the logits (145.9 MB > L2).
    Returns (us per call, bytes per call)."""
    from paper_2606_31160_gb300 import sd, workloads
    w = workloads.stochastic()
    B_, K_, V_ = w["B"], w["K"], w["V"]
    sets = [(w["z_target"].to(device), w["z_draft"].to(device)) for _ in range(2)]
    dr, u = w["draft"].to(device), w["u"].to(device)
    ws = sd.workspace(sd.sample_workspace_bytes(B_, K_, V_), device)
    n_emit = torch.zeros(B_, dtype=torch.int32, device=device)
    tokens = torch.zeros((B_, K_ + 1), dtype=torch.int32, device=device)

    def calls():
        for i in range(2 * reps):
            zt, zd = sets[i % 2]
            sd.accept_sample(zt, zd, dr, u, w["temperature"], ws=ws, n_emit=n_emit, tokens=tokens)

    g = capture(calls)
    ms = time_graph(g, 5) / (2 * reps)
    nbytes = (B_ * (K_ + 1) * V_ + B_ * K_ * V_) * 4
    return ms * 1e3, nbytes


def time_draft_steps(device, reps=20):
    """The draft's propose loop for one attention layer (16 q / 4 KV heads x 128,
    L = 4096, FlatRoPE = M-RoPE at (m, m, m)): 7 single-row decode steps, each one
    sd_verify_layer call (rotation at m = L + s, append, attention over
    L + s + 1 keys), then the rollback to the committed length and the reset
    to L, in a graph. Returns us per step."""
    from paper_2606_31160_gb300 import sd, workloads
    w = workloads.draft_flat()
    L_, steps = w["L"], w["steps"]
    lens = torch.full((1,), L_, dtype=torch.int32, device=device)
    lens0 = lens.clone()
    cache = sd.KVCache(w["k_cache"].to(device), w["v_cache"].to(device), lens)
    q = [w["q"][s].to(device) for s in range(steps)]
    k = [w["k_new"][s].to(device) for s in range(steps)]
    v = [w["v_new"][s].to(device) for s in range(steps)]
    pos = [torch.full((1, 1, 3), L_ + s, dtype=torch.int32, device=device) for s in range(steps)]
    out = [torch.empty_like(x) for x in q]
    ws = sd.workspace(sd.layer_workspace_bytes(1, 1, 16, 4, 128, cache.shape[2]), device)
    committed = torch.tensor([w["committed"]], dtype=torch.int32, device=device)

    def loop():
        for s in range(steps):
            sd.verify_layer(q[s], k[s], v[s], pos[s], SECTIONS, cache, 0, w["base"], out=out[s], ws=ws)
        sd.kv_rollback(lens, committed, steps)
        lens.copy_(lens0, non_blocking=True)

    g = capture(loop)
    ms = time_graph(g, reps)
    assert sd.get_device_error() == 0
    return ms * 1e3 / steps


def time_tiny_step(device, reps=200):
    """The tiny verify step (B = 1, 4 q / 1 KV head, head_dim 64, L = 256 = 192
    vision patches + 64 text tokens, K = 4, M-RoPE sections [8,12,12]): one
    sd_verify_layer call (head_dim 64 runs M-RoPE, append and attention as three
    kernels), the greedy accept over fp32 logits [1][5][4096] and the rollback,
    then the length put back, in a graph of `reps` steps. A latency figure: the
    step moves ~0.1 MB. Returns us per step."""
    from paper_2606_31160_gb300 import sd, workloads
    case = workloads.tiny()
    R_ = case.R
    q, k, v, pos = (x.to(device) for x in (case.q, case.k_new, case.v_new, case.pos))
    lens = torch.from_numpy(case.prefix.astype(np.int32)).to(device)
    lens0 = lens.clone()
    cache = sd.KVCache(case.k_cache.to(device), case.v_cache.to(device), lens)
    logits, draft = case.extra["logits"].to(device), case.extra["draft"].to(device)
    ws = sd.workspace(sd.greedy_workspace_bytes(1, R_ - 1, logits.shape[-1]), device)
    ws_l = sd.workspace(sd.layer_workspace_bytes(1, R_, case.Hq, case.Hkv, case.D, case.cap), device)
    out = torch.empty_like(q)
    n_emit = torch.zeros(1, dtype=torch.int32, device=device)
    tokens = torch.zeros((1, R_), dtype=torch.int32, device=device)
    argmax = torch.zeros((1, R_), dtype=torch.int32, device=device)

    def steps():
        for _ in range(reps):
            sd.verify_layer(q, k, v, pos, case.sections, cache, case.interleaved, case.base, out=out, ws=ws_l)
            sd.accept_greedy(logits, draft, ws=ws, n_emit=n_emit, tokens=tokens, argmax=argmax)
            sd.kv_rollback(lens, n_emit, R_)
            lens.copy_(lens0, non_blocking=True)

    g = capture(steps)
    ms = time_graph(g, 5)
    assert sd.get_device_error() == 0
    return ms * 1e3 / reps


def time_stochastic_step(device, layers=LAYERS):
    """The stochastic-acceptance step: 36 fused target layers at B = 8 (L = 4096,
    R = 8, 32 q / 8 KV x 128, one cache per layer: 4.84 GB streamed from HBM),
    then rejection sampling over fp32 logits [8][8][151936] (T = 0.6) and the
    rollback of all 36 lengths to the sampled commits, in a graph. Caches and
    rows ~ N(0, 1) bf16 from a seeded device generator. Returns (us per step,
    algorithmic bytes per step)."""
    from paper_2606_31160_gb300 import sd, workloads
    B_ = 8
    gen = torch.Generator(device=device)
    gen.manual_seed(5000)
    cap = L + R

    def normal(*shape):
        return torch.randn(shape, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)

    lens = torch.full((layers, B_), L, dtype=torch.int32, device=device)
    lens0 = lens.clone()
    caches, qs, ks, vs, outs, wss = [], [], [], [], [], []
    for l in range(layers):
        kc = torch.zeros((B_, HKV, cap, D), dtype=torch.bfloat16, device=device)
        vc = torch.zeros_like(kc)
        kc[:, :, :L] = normal(B_, HKV, L, D)
        vc[:, :, :L] = normal(B_, HKV, L, D)
        caches.append(sd.KVCache(kc, vc, lens[l]))
        qs.append(normal(B_, R, HQ, D))
        ks.append(normal(B_, R, HKV, D))
        vs.append(normal(B_, R, HKV, D))
        outs.append(torch.empty_like(qs[-1]))
        wss.append(sd.workspace(sd.layer_workspace_bytes(B_, R, HQ, HKV, D, cap), device))
    qpos = torch.from_numpy(np.stack([workloads.text_positions(544, R)] * B_)).to(device)
    w = workloads.stochastic()
    zt, zd, dr, u = (w["z_target"].to(device), w["z_draft"].to(device), w["draft"].to(device), w["u"].to(device))
    ws_s = sd.workspace(sd.sample_workspace_bytes(B_, K, V), device)
    n_emit = torch.zeros(B_, dtype=torch.int32, device=device)
    tokens = torch.zeros((B_, R), dtype=torch.int32, device=device)

    def step():
        for l in range(layers):
            sd.verify_layer(qs[l], ks[l], vs[l], qpos, SECTIONS, caches[l], 0, BASE, out=outs[l], ws=wss[l],
                            early=l > 0)
        sd.accept_sample(zt, zd, dr, u, w["temperature"], ws=ws_s, n_emit=n_emit, tokens=tokens)
        sd.kv_rollback(lens, n_emit, R)
        lens.copy_(lens0, non_blocking=True)

    g = capture(step)
    ms = time_graph(g, 10)
    assert sd.get_device_error() == 0
    logits = (B_ * R * V + B_ * K * V) * 4
    del caches, qs, ks, vs, outs, wss
    torch.cuda.empty_cache()
    return ms * 1e3, layers * layer_bytes(B_) + logits  # the same accounting as the main step


def time_long_draft_step(device, K_=16, layers=LAYERS):
    """The verify step of a block-diffusion draft (Sec. 5: blocks of K = 16
    tokens): 36 fused target layers at B = 1, L = 4096, R = 17 (68 packed rows
    per KV head: two 64-row m-blocks), one cache per layer, then the greedy
    accept over bf16 logits [1][17][151936] and the rollback, in a graph.
    Returns (us per step, algorithmic bytes per step)."""
    from paper_2606_31160_gb300 import sd, workloads
    R_ = K_ + 1
    gen = torch.Generator(device=device)
    gen.manual_seed(6000)
    cap = L + R_

    def normal(*shape):
        return torch.randn(shape, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)

    lens = torch.full((layers, 1), L, dtype=torch.int32, device=device)
    lens0 = lens.clone()
    caches, qs, ks, vs, outs, wss = [], [], [], [], [], []
    for l in range(layers):
        kc = torch.zeros((1, HKV, cap, D), dtype=torch.bfloat16, device=device)
        vc = torch.zeros_like(kc)
        kc[:, :, :L] = normal(1, HKV, L, D)
        vc[:, :, :L] = normal(1, HKV, L, D)
        caches.append(sd.KVCache(kc, vc, lens[l]))
        qs.append(normal(1, R_, HQ, D))
        ks.append(normal(1, R_, HKV, D))
        vs.append(normal(1, R_, HKV, D))
        outs.append(torch.empty_like(qs[-1]))
        wss.append(sd.workspace(sd.layer_workspace_bytes(1, R_, HQ, HKV, D, cap), device))
    qpos = torch.from_numpy(workloads.text_positions(544, R_)[None]).to(device)
    logits = normal(1, R_, V)
    draft = torch.randint(0, V, (1, K_), generator=gen, device=device, dtype=torch.int32)
    ws_g = sd.workspace(sd.greedy_workspace_bytes(1, K_, V), device)
    n_emit = torch.zeros(1, dtype=torch.int32, device=device)
    tokens = torch.zeros((1, R_), dtype=torch.int32, device=device)
    argmax = torch.zeros((1, R_), dtype=torch.int32, device=device)

    def step():
        for l in range(layers):
            sd.verify_layer(qs[l], ks[l], vs[l], qpos, SECTIONS, caches[l], 0, BASE, out=outs[l], ws=wss[l],
                            early=l > 0)
        sd.accept_greedy(logits, draft, ws=ws_g, n_emit=n_emit, tokens=tokens, argmax=argmax)
        sd.kv_rollback(lens, n_emit, R_)
        lens.copy_(lens0, non_blocking=True)

    g = capture(step)
    ms = time_graph(g, 20)
    assert sd.get_device_error() == 0
    rows = 2 * R_ * (2 * HQ + 3 * HKV) * D  # q in / out, rotated q, new k / v rows, out (as layer_bytes)
    nbytes = layers * (L * HKV * D * 2 * 2 + rows) + R_ * V * 2
    del caches, qs, ks, vs, outs, wss
    torch.cuda.empty_cache()
    return ms * 1e3, nbytes


def oracle_layer_sample(case, logits, draft):
    """The float64 oracle on one layer of the step plus the acceptance:
    returns bytes of the workload it covered (same accounting as the GPU)."""
    import oracle
    f64 = lambda t: t.float().numpy().astype(np.float64)
    pos = case.pos.numpy()[:, :, None, :]
    q = oracle.mrope_apply(f64(case.q), pos, SECTIONS, 0, BASE)
    k = oracle.mrope_apply(f64(case.k_new), pos, SECTIONS, 0, BASE)
    kc, vc, lens = oracle.kv_append(f64(case.k_cache), f64(case.v_cache), case.prefix, k, f64(case.v_new))
    oracle.verify_attention(q, kc, vc, lens)
    n_emit, _, _ = oracle.accept_greedy(f64(logits), draft.numpy())
    oracle.kv_rollback(lens, n_emit, R)
    return layer_bytes(1) + (step_bytes(1) - LAYERS * layer_bytes(1))


def host_cores():
    """Cores this process may run on (its affinity mask)."""
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS",
               "NUMEXPR_NUM_THREADS", "VECLIB_MAXIMUM_THREADS")


def time_oracle(budget_s, max_layers=None):
    """Oracle leg: whole layers of the step (rope, append, attention) plus the
    acceptance and rollback, repeated until budget_s is spent."""
    from paper_2606_31160_gb300 import workloads
    case = workloads.target_layer(B=1, layer=0, ell=[3])
    logits, draft = case.extra["logits"], case.extra["draft"]
    done_bytes, t0, n = 0, time.perf_counter(), 0
    while True:
        done_bytes += oracle_layer_sample(case, logits, draft)
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s or (max_layers and n >= max_layers):
            break
    return done_bytes / el / 1e9, n, el


def time_oracle_threads(budget_s, threads):
    """The oracle leg in a fresh interpreter whose BLAS / OpenMP pools are capped
    at `threads` (the variables must be set before numpy loads, hence a child
    process). Returns (GB/s, layers, seconds)."""
    env = dict(os.environ)
    for v in THREAD_VARS:
        env[v] = str(threads)
    out = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-leg", "--cpu-budget", str(budget_s)],
                         env=env, capture_output=True, text=True, timeout=budget_s * 4 + 300)
    if out.returncode != 0:
        raise RuntimeError("oracle leg failed:\n" + out.stderr[-2000:])
    d = json.loads(out.stdout.strip().splitlines()[-1])
    return d["gbs"], d["layers"], d["seconds"]


def oracle_leg(args):
    """Child-process entry of time_oracle_threads: one JSON line."""
    gbs, n, el = time_oracle(args.cpu_budget)
    print(json.dumps({"gbs": gbs, "layers": n, "seconds": el}), flush=True)


def cpu_baseline_pair(budget_s):
    """The oracle timed at 1 thread and at every core of the affinity mask."""
    cores = host_cores()
    one = time_oracle_threads(budget_s, 1)
    every = time_oracle_threads(budget_s, cores)
    return cores, one, every


# ------------------------------------------------------------------ main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-budget", type=float, default=10.0,
                    help="seconds of oracle time per leg (rank 0; two legs: 1 thread, all cores)")
    ap.add_argument("--oracle-leg", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--sweep", action="store_true",
                    help="time sd_verify_attention over the batched sweep grid (B x L x K) and "
                         "print one JSON line per point; prints no bench line")
    ap.add_argument("--sweep-b", type=int, nargs="*", default=None, help="restrict the sweep's batch sizes")
    ap.add_argument("--sweep-l", type=int, nargs="*", default=None, help="restrict the sweep's prefix lengths")
    ap.add_argument("--sweep-k", type=int, nargs="*", default=None, help="restrict the sweep's draft lengths")
    ap.add_argument("--floor", action="store_true",
                    help="measure the platform floors of the chained layers (empty dependent launches, "
                         "TMA streams of one layer's bytes) and print one JSON line per point; no bench line")
    ap.add_argument("--only", choices=["attention", "layer", "accept", "step", "sample", "tiny"], default=None,
                    help="profiling mode: run one kernel family eagerly `steps` times on the "
                         "target-layer workload (sample: the stochastic-acceptance workload) "
                         "for ncu captures; prints no bench line")
    args = ap.parse_args()
    world, rank, local = dist_env()
    if args.warmup < 3:
        args.warmup = 3

    if args.oracle_leg:
        return oracle_leg(args)
    if args.impl == "reference":
        return reference_arm(args, world, rank)
    if args.only:
        return profile_only(args)
    if args.sweep:
        return sweep(args)
    if args.floor:
        return floor(args)

    import torch.distributed as dist
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=device)

    from paper_2606_31160_gb300 import build, sd
    build.build()
    sd.lib()

    st = Step(device, scene=scenes_of_rank(1, rank)[0])
    # eager warm-up (sets kernel attributes before any capture), then graphs
    for _ in range(2):
        st.run()
    torch.cuda.synchronize()
    st.run_unfused()
    for l in range(LAYERS):  # the standalone attention needs the appended rows
        sd.kv_append(st.caches[l], st.k[l], st.v[l])
    g_attn = capture(st.attention_only)
    g_attn_plain = capture(lambda: st.attention_only(early=False))
    st.lens.copy_(st.lens0)
    torch.cuda.synchronize()
    g_step = capture(st.run)
    g_layers = capture(st.layers_only)
    g_unfused = capture(st.run_unfused)
    g_acc = capture(st.accept_chain)
    for _ in range(args.warmup):
        g_step.replay()
    torch.cuda.synchronize()
    assert sd.get_device_error() == 0

    # ---- timed region: K whole steps
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        e0.record(stream)
        for _ in range(args.steps):
            g_step.replay()
        e1.record(stream)
        e1.synchronize()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms_total = max_over_ranks(e0.elapsed_time(e1), world, device)
    ms_step = ms_total / args.steps

    # ---- dominant kernel: the fused verify layer, its 36 launches alone
    #      (distinct caches, chained as programmatic dependent launches)
    reps = max(20, min(2000, args.steps))
    ms_layer_launch = time_graph(g_layers, reps) / LAYERS
    ms_accept = time_graph(g_acc, max(5, reps // Step.ACCEPT_COPIES)) / Step.ACCEPT_COPIES
    ms_unfused = time_graph(g_unfused, max(20, min(500, args.steps)))
    # the standalone attention kernel over appended caches, for reference
    for l in range(LAYERS):
        sd.kv_append(st.caches[l], st.k[l], st.v[l])
    ms_attn_launch = time_graph(g_attn, reps) / LAYERS
    ms_attn_plain = time_graph(g_attn_plain, reps) / LAYERS
    # the attention-budget diagnostic (Table tab:attn-budget) on the same 36
    # appended caches: visual keys = the 4 cameras' 896 patches each
    nvis = torch.full((1,), 4 * 896, dtype=torch.int32, device=device)
    mass = torch.empty((1, R, HQ, 3), dtype=torch.float32, device=device)
    ent = torch.empty((1, R, HQ), dtype=torch.float32, device=device)
    g_budget = capture(lambda: [sd.attention_budget(st.q[l], st.caches[l], nvis, mass=mass, entropy=ent)
                                for l in range(LAYERS)])
    ms_budget = time_graph(g_budget, reps) / LAYERS
    st.lens.copy_(st.lens0)
    torch.cuda.synchronize()
    # ---- the small kernels of the path, per call: M-RoPE of one layer's rows,
    #      the rollback of all 36 lengths (committed = R: lengths unchanged), and
    #      one layer's append (timed with a rollback of the same R rows that puts
    #      its length back; the rollback alone is subtracted)
    full = torch.full((1,), R, dtype=torch.int32, device=device)
    zero = torch.zeros(1, dtype=torch.int32, device=device)
    g_rope = capture(lambda: [sd.rope_apply(st.q[l], st.k[l], st.pos, SECTIONS, 0, BASE) for l in range(LAYERS)])
    g_rb = capture(lambda: [sd.kv_rollback(st.lens, full, R) for _ in range(LAYERS)])
    g_ap = capture(lambda: [(sd.kv_append(st.caches[l], st.k[l], st.v[l]), sd.kv_rollback(st.lens[l], zero, R))
                            for l in range(LAYERS)])
    ms_rope = time_graph(g_rope, reps) / LAYERS
    ms_rollback = time_graph(g_rb, reps) / LAYERS
    ms_append = time_graph(g_ap, reps) / LAYERS - ms_rollback
    st.d_in.copy_(st.h_in)  # the rotations above changed the q / k rows in place
    st.lens.copy_(st.lens0)
    torch.cuda.synchronize()
    assert sd.get_device_error() == 0

    # ---- end to end: pinned host inputs -> device, step, result -> host
    e2e_steps = max(10, min(500, args.steps))
    for _ in range(3):
        st.h2d(); g_step.replay(); st.d2h()
    torch.cuda.synchronize()
    a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a0.record(stream)
    for _ in range(e2e_steps):
        st.h2d()
        g_step.replay()
        st.d2h()
    a1.record(stream)
    a1.synchronize()
    ms_e2e = max_over_ranks(a0.elapsed_time(a1) / e2e_steps, world, device)
    assert sd.get_device_error() == 0
    # the stochastic-acceptance workload (rejection sampling over B = 8 scenes),
    # its whole step (36 layers at B = 8 + sampling), and the draft's propose loop
    sample_us, sample_bytes = time_sample_accept(device) if rank == 0 else (None, None)
    draft_us = time_draft_steps(device) if rank == 0 else None
    tiny_us = time_tiny_step(device) if rank == 0 else None
    stoch_us, stoch_bytes = time_stochastic_step(device) if rank == 0 else (None, None)
    long_us, long_bytes = time_long_draft_step(device) if rank == 0 else (None, None)
    assert sd.get_device_error() == 0

    if rank != 0:
        if world > 1:
            dist.barrier()
            dist.destroy_process_group()
        return

    peak, peak_kind = measured_peaks()
    value = aggregate_gbs(step_bytes(1), world, ms_step)
    achieved = layer_bytes(1) / (ms_layer_launch * 1e-3) / 1e9
    traffic = ncu_traffic()
    cores, (one_gbs, one_layers, one_s), (all_gbs, all_layers, all_s) = cpu_baseline_pair(args.cpu_budget)
    line = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_step, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded Philox; no clips or weights exist here)",
        "config": {
            "workload": "8B-class target verify step: 36 layers x (M-RoPE + KV append + verify attention, "
                        "L=4096, K=7, 32q/8kv x 128, bf16) + greedy accept over bf16 logits V=151936 + rollback",
            "batch_per_gpu": 1, "layers": LAYERS, "prefix_len": L, "K": K, "q_heads": HQ, "kv_heads": HKV,
            "head_dim": D, "vocab": V, "mrope_section": list(SECTIONS), "rope_base": BASE,
            "parallelism": "replicas" if world > 1 else "single-gpu",
            "l2": "inputs larger than L2: 36 distinct KV caches (605 MB) streamed per step",
            "timing": "CUDA graph of one step, replayed; CUDA events on the launching stream",
            "layer_kernel": "fused M-RoPE + KV append + verify attention per layer (sd_verify_layer)",
        },
        "verify_step_us": round(ms_step * 1e3, 3),
        "per_layer_us": round(ms_step * 1e3 / LAYERS, 3),
        "layer_us": round(ms_layer_launch * 1e3, 3),
        "attention_us": round(ms_attn_launch * 1e3, 3),
        "attention_us_no_early_prefix": round(ms_attn_plain * 1e3, 3),
        "budget_us": round(ms_budget * 1e3, 3),
        "unfused_verify_step_us": round(ms_unfused * 1e3, 3),
        "rope_us": round(ms_rope * 1e3, 3),
        "kv_append_us": round(ms_append * 1e3, 3),
        "kv_rollback_us": round(ms_rollback * 1e3, 3),
        "accept_us": round(ms_accept * 1e3, 3),
        "sample_accept_us": round(sample_us, 3),
        "sample_accept_gbs": round(sample_bytes / (sample_us * 1e-6) / 1e9, 1),
        "draft_step_us": round(draft_us, 3),
        "tiny_step_us": round(tiny_us, 3),
        "stochastic_step_us": round(stoch_us, 2),
        "stochastic_step_gbs": round(stoch_bytes / (stoch_us * 1e-6) / 1e9, 1),
        "block_draft_step_us": round(long_us, 2),
        "block_draft_step_gbs": round(long_bytes / (long_us * 1e-6) / 1e9, 1),
        "bytes_per_step": step_bytes(1),
        "roofline": {
            "kernel": "sd_verify_layer -> verify_attn_tc_kernel<fused> (M-RoPE + append + attention, tcgen05)",
            "bound": "hbm",
            "achieved": round(achieved, 1),
            "peak": peak,
            "peak_kind": peak_kind,
            "unit": "GB/s",
            "frac": round(achieved / peak, 4),
            "traffic": traffic,
            "algorithmic_bytes_per_launch": layer_bytes(1),
            "timing": "36 chained launches of the layer kernel in one graph; average = total / 36",
        },
        "cpu_baseline": {
            "value": round(all_gbs, 4),
            "unit": "GB/s",
            "cores": cores,
            "kind": "oracle",
            "sample": "%d full target layers (M-RoPE, append, attention over 4104 keys, all 32 heads) each "
                      "with the greedy accept over 8 x 151936 and the rollback, float64 numpy, %.1f s, BLAS and "
                      "OpenMP pools at %d threads (the affinity mask)" % (all_layers, all_s, cores),
            "one_thread": {"value": round(one_gbs, 4), "unit": "GB/s", "cores": 1,
                           "sample": "%d layers in %.1f s, every pool at 1 thread" % (one_layers, one_s)},
        },
        "e2e": {
            "value": round(aggregate_gbs(step_bytes(1), world, ms_e2e), 2),
            "unit": "GB/s",
            "ms_per_step": round(ms_e2e, 5),
            "h2d_bytes_per_step": st.h2d_bytes,
            "d2h_bytes_per_step": st.d2h_bytes,
        },
        "gpu_launches": args.steps * (LAYERS + 2),
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


SWEEP_B, SWEEP_L, SWEEP_K = (1, 8, 32), (2048, 4096, 8192, 16384), (1, 2, 4, 8, 16)


def sweep(args):
    """sd_verify_attention over the batched sweep (B scenes, ragged L_b ~
    U[0.75 L, L], 32 q / 8 KV x 128, bf16): per point, the rotated rows are
    appended and the attention launch is timed in a CUDA graph over enough
    distinct caches that one replay streams > 2 x L2 (inputs larger than L2).
    Algorithmic bytes: K and V of every key (L_b + R per scene and KV head),
    plus Q read and O written."""
    from paper_2606_31160_gb300 import build, sd, workloads
    build.build()
    sd.lib()
    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    peak, peak_kind = measured_peaks()
    l2_bytes = 129 * 2 ** 20
    for B in args.sweep_b or SWEEP_B:
        for Lp in args.sweep_l or SWEEP_L:
            for Kp in args.sweep_k or SWEEP_K:
                R_ = Kp + 1
                prefix, q, k_new, v_new, pos, kc, vc, cap = workloads.sweep_case_device(B, Lp, Kp, device)
                nbytes = int(sum(int(p) + R_ for p in prefix)) * HKV * D * 2 * 2 + 2 * B * R_ * HQ * D * 2
                copies = max(1, min(64, -(-(2 * l2_bytes) // nbytes)))
                lens = torch.from_numpy(np.asarray(prefix, dtype=np.int32)).to(device)
                sd.rope_apply(q, k_new, pos, SECTIONS, 0, BASE)
                caches = []
                for c in range(copies):
                    cache = sd.KVCache(kc if c == 0 else kc.clone(), vc if c == 0 else vc.clone(), lens.clone())
                    sd.kv_append(cache, k_new, v_new)
                    caches.append(cache)
                del kc, vc
                outs = [torch.empty_like(q) for _ in range(copies)]
                ws = [sd.workspace(sd.attention_workspace_bytes(B, R_, HQ, HKV, D, cap), device)
                      for _ in range(copies)]

                def launches():
                    for c in range(copies):
                        sd.verify_attention(q, caches[c], out=outs[c], ws=ws[c])

                g = capture(launches)
                ms_one = time_graph(g, 3) / copies
                reps = max(5, min(2000, int(100.0 / max(ms_one * copies, 1e-3))))
                ms = time_graph(g, reps) / copies
                gbs = nbytes / (ms * 1e-3) / 1e9
                assert sd.get_device_error() == 0
                print(json.dumps({"sweep": {"B": B, "L": Lp, "K": Kp, "sum_keys": int(sum(prefix)) + B * R_,
                                            "us": round(ms * 1e3, 3), "gbs": round(gbs, 1),
                                            "frac": round(gbs / peak, 4), "peak": peak, "peak_kind": peak_kind,
                                            "bytes": nbytes, "copies": copies}}), flush=True)
                del caches, outs, ws, g
                torch.cuda.empty_cache()


# The 32-row fused layer kernel's launch shape: 8 heads x a cluster of 8 CTAs
# of 352 threads, 230,976 bytes of dynamic shared memory, 256 tensor-memory
# columns.
FLOOR_SHAPE = {"ctas": 64, "cluster": 8, "threads": 352, "smem": 230976, "tmem_cols": 256}


def floor(args):
    """Platform floors of the chained verify layers (one JSON line each, no
    bench line). (1) A chain of 36 launches that do no work, in the fused
    layer kernel's launch shape, each a programmatic dependent launch of the
    one before (or plain launches): the release latency that every chained
    layer pays. (2) A chain of 36 launches that only stream one target layer's
    bytes (17,170,432 B as rows of 256 B, a distinct slice per launch, 618 MB
    in all: larger than L2) through shared memory by TMA, over 64 to 304 CTAs,
    with the dependency wait at the start, after the first ring fill (as the
    layer kernel's early prefix), at the end, or no dependent launch at all.
    CUDA events around graph replays on the floor library's own stream."""
    import ctypes
    from paper_2606_31160_gb300 import build
    build.build()
    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    torch.cuda.init()
    lib = ctypes.CDLL(build.FLOOR_LIB)
    lib.sdfloor_empty_chain.restype = ctypes.c_int
    lib.sdfloor_empty_chain.argtypes = [ctypes.c_int] * 8 + [ctypes.POINTER(ctypes.c_float)]
    lib.sdfloor_stream_chain.restype = ctypes.c_int
    lib.sdfloor_stream_chain.argtypes = [ctypes.c_void_p, ctypes.c_longlong, ctypes.c_int, ctypes.c_int,
                                         ctypes.c_int, ctypes.c_int, ctypes.POINTER(ctypes.c_float)]
    peak, peak_kind = measured_peaks()
    us = ctypes.c_float(0.0)
    sh = FLOOR_SHAPE
    for pdl in (1, 0):
        for tmem in (sh["tmem_cols"], 0):
            rc = lib.sdfloor_empty_chain(LAYERS, sh["ctas"], sh["cluster"], sh["threads"], sh["smem"], tmem, pdl,
                                         200, ctypes.byref(us))
            print(json.dumps({"floor": "empty", "layers": LAYERS, "ctas": sh["ctas"], "cluster": sh["cluster"],
                              "threads": sh["threads"], "smem": sh["smem"], "tmem_cols": tmem, "pdl": pdl,
                              "us_per_launch": round(us.value, 3), "rc": rc}), flush=True)
    nbytes = layer_bytes()
    rows = nbytes // 256
    buf = torch.zeros(LAYERS * rows * 128, dtype=torch.bfloat16, device=device)
    torch.cuda.synchronize()
    names = {-1: "no dependent launch", 0: "wait at start", 1: "wait after first ring fill", 2: "wait at end"}
    for ctas in (64, 128, 152, 304):
        for waitpos in (-1, 0, 1, 2):
            rc = lib.sdfloor_stream_chain(ctypes.c_void_p(buf.data_ptr()), rows, LAYERS, ctas, waitpos, 50,
                                          ctypes.byref(us))
            gbs = nbytes / (us.value * 1e-6) / 1e9 if us.value > 0 else 0.0
            print(json.dumps({"floor": "stream", "layers": LAYERS, "bytes_per_launch": nbytes, "ctas": ctas,
                              "wait": names[waitpos], "us_per_launch": round(us.value, 3), "gbs": round(gbs, 1),
                              "frac": round(gbs / peak, 4), "peak": peak, "peak_kind": peak_kind, "rc": rc}),
                  flush=True)
    err = lib.sdfloor_take_error()
    print(json.dumps({"floor": "done", "device_error": err}), flush=True)
    return 0 if err == 0 else 1


def profile_only(args):
    """Eager launches of one kernel family on the 36-layer target workload,
    for profiler captures (a handful of launches, no timing output)."""
    from paper_2606_31160_gb300 import build, sd, workloads
    build.build()
    torch.cuda.set_device(0)
    if args.only == "sample":
        # sd_accept_sample on the stochastic-acceptance workload (B=8, K=7, V=151936)
        dev = torch.device("cuda", 0)
        w = workloads.stochastic()
        zt, zd = w["z_target"].to(dev), w["z_draft"].to(dev)
        dr, u = w["draft"].to(dev), w["u"].to(dev)
        ws = sd.workspace(sd.sample_workspace_bytes(w["B"], w["K"], w["V"]), dev)
        for _ in range(args.steps):
            sd.accept_sample(zt, zd, dr, u, w["temperature"], ws=ws)
        torch.cuda.synchronize()
        print(json.dumps({"profile_only": args.only, "launches": args.steps,
                          "device_error": sd.get_device_error()}))
        return
    if args.only == "tiny":
        # the tiny verify step (4 q / 1 KV x 64, L = 256, K = 4): M-RoPE, append
        # and the mma.sync attention kernel (head_dim 64), accept, rollback
        dev = torch.device("cuda", 0)
        case = workloads.tiny()
        q, k, v, pos = (x.to(dev) for x in (case.q, case.k_new, case.v_new, case.pos))
        lens = torch.from_numpy(case.prefix.astype(np.int32)).to(dev)
        cache = sd.KVCache(case.k_cache.to(dev), case.v_cache.to(dev), lens)
        logits, draft = case.extra["logits"].to(dev), case.extra["draft"].to(dev)
        for _ in range(args.steps):
            lens.copy_(torch.from_numpy(case.prefix.astype(np.int32)).to(dev))
            sd.verify_layer(q, k, v, pos, case.sections, cache, case.interleaved, case.base)
            n_emit, tokens, _ = sd.accept_greedy(logits, draft)
        torch.cuda.synchronize()
        print(json.dumps({"profile_only": args.only, "launches": args.steps,
                          "device_error": sd.get_device_error()}))
        return
    st = Step(torch.device("cuda", 0))
    st.run()  # one full step: rope, append, attention, accept, rollback
    torch.cuda.synchronize()
    for l in range(LAYERS):  # leave every cache holding L + R keys
        sd.kv_append(st.caches[l], st.k[l], st.v[l])
    for i in range(args.steps):
        if args.only == "attention":
            sd.verify_attention(st.q[i % LAYERS], st.caches[i % LAYERS], out=st.out[i % LAYERS])
        elif args.only == "layer":
            l = i % LAYERS
            st.lens[l].fill_(L)
            sd.verify_layer(st.q[l], st.k[l], st.v[l], st.pos, SECTIONS, st.caches[l], 0, BASE,
                            out=st.out[l], ws=st.ws_layer[l])
        elif args.only == "accept":
            st.accept_only()
        else:
            st.lens.fill_(L)
            st.run()
    torch.cuda.synchronize()
    print(json.dumps({"profile_only": args.only, "launches": args.steps,
                      "device_error": sd.get_device_error()}))


def reference_arm(args, world, rank):
    """The float64 oracle run as the reference arm on the host cores: each
    step is one full layer of the workload plus the acceptance and rollback."""
    if rank != 0:
        return
    from paper_2606_31160_gb300 import workloads
    case = workloads.target_layer(B=1, layer=0, ell=[3])
    logits, draft = case.extra["logits"], case.extra["draft"]
    for _ in range(args.warmup):
        oracle_layer_sample(case, logits, draft)
    steps = min(args.steps, 50)
    t0 = time.perf_counter()
    done = 0
    for _ in range(steps):
        done += oracle_layer_sample(case, logits, draft)
    el = time.perf_counter() - t0
    value = done / el / 1e9
    line = {
        "impl": "reference",
        "metric": METRIC,
        "value": round(value, 4),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": steps,
        "warmup": args.warmup,
        "ms_per_step": round(el / steps * 1e3, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic (seeded Philox)",
        "config": {"workload": "8B-class target verify step, one layer per step (sample): M-RoPE + append + "
                               "attention L=4096 K=7 32q/8kv x 128 + greedy accept V=151936 + rollback",
                   "parallelism": "host cores"},
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": host_cores(), "kind": "oracle",
                         "sample": "one target layer + acceptance per step, %d steps, numpy's default "
                                   "BLAS pool over the affinity mask" % steps},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
