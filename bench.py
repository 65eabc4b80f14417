#!/usr/bin/env python
"""Throughput benchmark of the GB300 DLM compressor (one JSON line on stdout).

Headline workload (the largest single-GPU configuration): an 8B-shaped masked
bf16 DLM (32 layers, d = 4096, 32 heads of 128, FFN 12288, V = 126464,
random-init N(0, 0.02)) coding 2^20 seeded Zipf(1.05)-bigram tokens in
windows of 1024 tokens, 512 windows per batch, top-16 positions per step by
confidence over the whole window (64 denoising steps per window), 24-bit
integer CDFs.

One benchmark step = one denoising step of compression plus the matching
denoising step of decompression over a whole batch (512 windows x 1024
tokens): the forward pass of the batch, the LM head and quantiser on the
candidate rows (the still-masked positions), selection, and coding
(decoding) of 16 tokens per window.  The encoder runs W + K + 1 denoising steps
of the batch and terminates its streams; the decoder then replays the same
W + K + 1 steps from those streams and must reproduce the encoder's state.
The first W steps of each direction are warm-up, the next K are timed (CUDA
events on the library's stream, device synchronised around each timed
segment), and one more untimed step per direction records CUDA events
around every launch for the per-kernel split and the rooflines.  ``value`` =
input bytes coded (and decoded) per step x K / the summed time; compress and
decompress are also reported separately.

``secondary`` holds the small byte-level workload (8 layers, d = 512, V =
256; one 512 KiB batch compressed and decompressed per step), a timed prefix
of the 7B GQA-shaped entropy-schedule workload (64 windows of 2048 tokens,
V = 152064; two denoising steps each way) and the
isolated quantise + select workload (65536 x 126464 float32 logits, 24-bit
CDFs plus scores, top-32 of groups of 1024) at full size.

``--impl reference`` times the CPU oracle (oracle/) instead, on a bounded
sample of the headline workload.  Under torchrun each rank codes its own
batch (weak scaling, no collective on the data path).
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "input bytes/sec compress+decompress on 1 GB300; bits/byte; % of roofline"
C4 = dict(n_layers=32, d=4096, n_heads=32, n_kv_heads=32, ffn=12288, vocab=126464, seed=0)
C4_TOKENS, C4_CHUNK, C4_BATCH, C4_K = 1 << 20, 1024, 512, 16
PROF_STEPS = 1  # untimed denoising steps per direction whose launches carry events (the kernel split)
C4_WORKLOAD = ("8B-shaped masked DLM, bf16, random-init: 32 layers d=4096 32 heads (hd 128) FFN 12288 V=126464, "
               "bidirectional attention; 2^20 Zipf(1.05) bigram tokens, windows of 1024 tokens, 512 windows per "
               "batch, top-16 by confidence per step over the whole window, 24-bit CDFs")
C2 = dict(n_layers=8, d=512, n_heads=8, n_kv_heads=8, ffn=2048, vocab=256, seed=0)
C2_CHUNK, C2_BATCH, C2_BLOCK, C2_K, C2_INPUT = 512, 1024, 128, 8, 4 << 20
C2_WORKLOAD = ("small byte-level masked DLM, bf16, 8 layers d=512 8 heads FFN 2048 V=256; 4 MiB order-2 "
               "Markov/Zipf(1.1) bytes; windows of 512 B, 1024 windows per batch, block 128, top-k 8 by "
               "confidence, 16-bit CDFs")
C3_ROWS, C3_V, C3_GROUP, C3_TOPK = 65536, 126464, 1024, 32
# Mean DRAM bytes per tcgen05 GEMM launch of an 8B-shaped layer at 512 windows, scaled from an ncu
# capture of the same kernels at 16 windows (B is re-read once per row group, so traffic grows with M)
GEMM_TRAFFIC_PER_LAUNCH = 53.4e9
CLASSES = ["gemm_tcgen05", "gemm_cuda_core", "attention", "quantize", "select", "code", "norm_rope_embed", "other"]


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        p = json.load(open(path))
        return p["hbm_gbs"], p["bf16_tflops"], p["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    return ws, int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0"))


def host_cores():
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms while running."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.out = open(os.path.join("/tmp", "dlmz_clocks_%d.csv" % os.getpid()), "w+")
            self.proc = subprocess.Popen(["nvidia-smi", "--query-gpu=" + self.Q, "--format=csv,noheader,nounits",
                                          "-lms", "200", "-i", str(self.idx)], stdout=self.out,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.out.seek(0)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.out.read().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        self.out.close()
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---- CPU oracle baseline ----------------------------------------------------------------------

class OracleSampler:
    """The CPU oracle on a bounded sample of one denoising step of the headline workload.

    set-up (untimed): the weights of one 8B-shaped layer, the embedding and the
    LM head (the oracle's own counter-based draws) and a 1024-token window of
    Zipf-bigram tokens with half of its positions masked.  sample(): one
    float64 transformer layer over the window (x 32 layers: they cost the same),
    the final norm, LM head and quantiser on 64 candidate rows (scaled to the
    520 candidate rows of an average step: 1024 masked positions at the first
    step, 16 at the last), selection of 16 and range coding of their symbols.
    Returns the extrapolated seconds per denoising step of one window.
    """

    def __init__(self):
        import numpy as np

        from oracle import model as OM
        from paper_2608_11249_gb300 import sources
        cfg = OM.ModelConfig(1, C4["d"], C4["n_heads"], C4["n_kv_heads"], C4["ffn"], C4["vocab"], "bf16",
                             seed=C4["seed"])
        t0 = time.perf_counter()
        self.w = OM.Weights(cfg, lazy=True)
        for which in range(7):
            self.w.layer(0, which)
        _ = self.w.embed, self.w.head
        self.init_s = time.perf_counter() - t0
        L, V = C4_CHUNK, C4["vocab"]
        self.tok = sources.zipf_bigram_tokens(L, V, seed=0).astype(np.int64)
        self.state = self.tok.copy()
        self.state[np.random.default_rng(0).random(L) < 0.5] = V

    def sample(self):
        import numpy as np

        from oracle import coder as OC
        from oracle import model as OM
        from oracle import quantizer as OQ
        from oracle import selector as OS
        from oracle import weights as OW
        w, V = self.w, C4["vocab"]
        t1 = time.perf_counter()
        h = OM.hidden(w, self.state)  # one layer, then the final norm
        t2 = time.perf_counter()
        rows = np.flatnonzero(self.state == V)[:64]
        logits = OW.round_f32(h[rows] @ w.head.T)
        P = OQ.precision_for_vocab(V)
        q = OQ.quantize(logits, P)
        t3 = time.perf_counter()
        pol = OS.Policy(kind=OS.TOPK_CONF, k=C4_K, block=0)
        sel = OS.select(np.ones(len(rows), dtype=bool), {i: q["W"][i] for i in range(len(rows))}, pol, 0)
        enc = OC.Encoder(P)
        for i in sel:
            sy = int(self.tok[rows[i]])
            enc.encode(int(q["cdf"][i, sy]), int(q["freq"][i, sy]))
        enc.finish()
        t4 = time.perf_counter()
        parts = {"layer_s": t2 - t1, "head_quant_s_per_520_rows": (t3 - t2) * 520.0 / len(rows),
                 "select_code_s": t4 - t3, "weight_init_s_excluded": self.init_s}
        per_step = C4["n_layers"] * parts["layer_s"] + parts["head_quant_s_per_520_rows"] + parts["select_code_s"]
        return per_step, parts


def oracle_child(threads):
    """Run oracle_sample_c4 in a child process with `threads` BLAS threads; return its JSON."""
    env = dict(os.environ)
    if threads:
        for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
            env[k] = str(threads)
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-child"], env=env, capture_output=True,
                       text=True, timeout=900)
    if r.returncode != 0:
        raise RuntimeError("oracle sample failed: " + r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def cpu_baseline(one_thread=False):
    """The oracle on the host cores: all cores (the figure) and, on request, one thread beside it."""
    cores = host_cores()
    allc = oracle_child(0)
    step_bytes = C4_K * 4  # one denoising step codes 16 tokens of 4 bytes per window
    val = step_bytes / (2.0 * allc["per_step_s"])  # compress + decompress each run the step
    out = {
        "value": val, "unit": "B/s", "cores": cores, "kind": "oracle",
        "sample": ("one denoising step of one 1024-token window of the headline workload, compress + decompress: "
                   "one float64 transformer layer timed x 32 layers, LM head + quantiser timed on 64 candidate "
                   "rows scaled to the 520 of an average step, selection + range coding of 16 symbols; "
                   "weight generation excluded; extrapolated"),
        "threads": "BLAS threads = all %d host cores (value); one thread (value_one_thread)" % cores,
        "seconds_per_window_step": allc["per_step_s"],
        "parts": allc["parts"],
    }
    if one_thread:  # the sample's wall time on one thread: under a minute on a Grace host
        one = oracle_child(1)
        out["value_one_thread"] = step_bytes / (2.0 * one["per_step_s"])
        out["seconds_per_window_step_one_thread"] = one["per_step_s"]
    return out


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    cores = host_cores()
    sampler = OracleSampler()
    vals, sample_s = [], []
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        per_step, _ = sampler.sample()
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            vals.append(C4_K * 4 / (2.0 * per_step))
            sample_s.append(dt)
    v = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "B/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * statistics.mean(sample_s),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded Zipf(1.05) bigram tokens); random-init N(0,0.02) weights",
            "config": {"workload": C4_WORKLOAD, "batch_chunks": C4_BATCH, "chunk_len": C4_CHUNK, "k": C4_K},
            "cpu_baseline": {"value": v, "unit": "B/s", "cores": cores, "kind": "oracle",
                             "sample": ("each step: one denoising step of one 1024-token window, compress + "
                                        "decompress, extrapolated from one float64 layer (x 32), the LM head + "
                                        "quantiser on 64 rows (scaled to 520) and selection + range coding of 16 "
                                        "symbols; ms_per_step is that sample's wall time; weight generation "
                                        "(%.0f s, once) excluded" % sampler.init_s)},
            "e2e": {"value": v, "unit": "B/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ---- GPU arms ---------------------------------------------------------------------------------

def _events():
    import torch
    return torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)


def _prof_add(acc, p):
    acc["launches"] += int(p.launches)
    for j in range(8):
        acc["n"][j] += int(p.n[j])
        acc["ms"][j] += float(p.ms[j])
        acc["flops"][j] += float(p.flops[j])
        acc["bytes"][j] += float(p.bytes[j])


def run_c4(args, dlmz, torch, rank, ws, dev):
    """The headline workload: K timed denoising steps each way over one batch (see the module docstring)."""
    import numpy as np
    from paper_2608_11249_gb300 import sources

    stream = torch.cuda.current_stream().cuda_stream
    V, L, nc, k = C4["vocab"], C4_CHUNK, C4_BATCH, C4_K
    m = dlmz.Model(C4["n_layers"], C4["d"], C4["n_heads"], C4["n_kv_heads"], C4["ffn"], V, dlmz.BF16, seed=C4["seed"])
    tokens = sources.zipf_bigram_tokens(C4_TOKENS, V, seed=0)
    n_batches = C4_TOKENS // (nc * L)
    b = rank % n_batches  # weak scaling: each rank its own batch of the input (cycling past the input's end)
    sym_h = tokens[b * nc * L:(b + 1) * nc * L].astype(np.int32).reshape(nc, L)
    sym = torch.from_numpy(sym_h).to(dev)
    state = torch.full((nc, L), V, dtype=torch.int32, device=dev)
    committed = torch.zeros(nc, dtype=torch.int32, device=dev)
    pol = dlmz.policy(dlmz.TOPK_CONF, k, 0)
    n_steps = args.warmup + args.steps + PROF_STEPS
    if n_steps * k > L:
        raise SystemExit("at most %d denoising steps per window" % (L // k))
    P = 24
    enc = dlmz.Coder(nc, L, V, P)
    enc.reset_encoder()
    clocks = ClockSampler(torch.cuda.current_device())
    prof_acc = {"launches": 0, "n": [0] * 8, "ms": [0.0] * 8, "flops": [0.0] * 8, "bytes": [0.0] * 8}

    def barrier():
        torch.cuda.synchronize()
        if ws > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    launches = [0]

    def phase(fn):
        """W untimed steps, K steps timed with events on the stream, then PROF_STEPS untimed steps with
        per-launch events for the kernel split (kept out of the timed region)."""
        for i in range(args.warmup):
            fn()
        barrier()
        n0 = dlmz.launch_count()
        e0, e1 = _events()
        e0.record()
        for i in range(args.steps):
            fn()
        e1.record()
        e1.synchronize()
        launches[0] += dlmz.launch_count() - n0
        barrier()
        prof = dlmz.Profile()
        dlmz.profile_begin()
        for i in range(PROF_STEPS):
            fn()
        dlmz.profile_end(prof)
        barrier()
        _prof_add(prof_acc, prof)
        return e0.elapsed_time(e1)

    clocks.start()
    enc_ms = phase(lambda: m.encode_step(enc, pol, 0, L, sym.data_ptr(), state.data_ptr(), committed.data_ptr(),
                                         stream))
    dlmz.check(stream)
    enc_state = state.clone()
    bits = torch.empty(nc, dtype=torch.int32, device=dev)
    cap = enc.capacity_units * 2
    raw = torch.zeros(nc * cap, dtype=torch.uint8, device=dev)
    enc.finish(bits.data_ptr(), raw.data_ptr(), 0, stream)
    dlmz.check(stream)
    offs = (torch.arange(nc, dtype=torch.int64, device=dev) * cap).contiguous()
    dec = dlmz.Coder(nc, L, V, P)
    dec.load_decoder(raw.data_ptr(), offs.data_ptr(), bits.data_ptr(), stream)
    state.fill_(V)
    dec_ms = phase(lambda: m.decode_step(dec, pol, 0, L, state.data_ptr(), committed.data_ptr(), stream))
    dlmz.check(stream)
    clk = clocks.stop()
    assert torch.equal(state, enc_state), "decoder state differs from the encoder's"
    revealed = int((enc_state != V).sum().item())
    assert revealed == nc * k * n_steps
    stream_bits = int(bits.to(torch.int64).sum().item())
    if ws > 1:
        from paper_2608_11249_gb300 import shard
        enc_ms = shard.max_over_ranks(enc_ms, device=dev)
        dec_ms = shard.max_over_ranks(dec_ms, device=dev)
    step_bytes = nc * k * 4  # input bytes (uint32 tokens) coded per denoising step of the batch
    total_ms = enc_ms + dec_ms
    value = ws * step_bytes * args.steps / (total_ms / 1000.0)
    enc.close()
    dec.close()
    del raw, bits, offs, state, sym, committed, enc_state

    # end to end through the host-buffer C ABI: whole files of 8 windows (the same model and policy;
    # host -> device copy of the input and device -> host copy of the result inside the timed region)
    e2e_nc = 8
    data = sources.tokens_to_bytes(tokens[:e2e_nc * L])
    e2e_steps = 1 if args.steps <= 3 else 2
    e2e_s, h2d, d2h = 0.0, 0, 0
    for i in range(e2e_steps):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        blob = m.compress(data, L, pol, e2e_nc)
        back = m.decompress(blob)
        torch.cuda.synchronize()
        e2e_s += time.perf_counter() - t0
        assert back == data
        h2d += len(data) + len(blob)
        d2h += len(blob) + len(back)
    e2e = {"value": ws * len(data) * e2e_steps / e2e_s, "unit": "B/s", "h2d_bytes_per_step": h2d // e2e_steps,
           "d2h_bytes_per_step": d2h // e2e_steps,
           "api": "dlmz_compress_ex + dlmz_decompress (host buffers), whole files of 8 windows x 1024 tokens "
                  "(128 denoising steps of forward over 8192 tokens each)",
           "bits_per_token": 8.0 * len(blob) / (len(data) / 4)}
    m.close()
    return {
        "value": value, "total_ms": total_ms, "enc_ms": enc_ms, "dec_ms": dec_ms, "step_bytes": step_bytes,
        "compress_Bps": ws * step_bytes * args.steps / (enc_ms / 1000.0),
        "decompress_Bps": ws * step_bytes * args.steps / (dec_ms / 1000.0),
        "bits_per_token_stream": stream_bits / float(revealed), "prof": prof_acc, "clocks": clk, "e2e": e2e,
        "launches": launches[0],
    }


C5 = dict(n_layers=28, d=3584, n_heads=28, n_kv_heads=4, ffn=18944, vocab=152064, seed=0)
C5_CHUNK, C5_BATCH, C5_TAU, C5_KMIN, C5_KMAX = 2048, 64, 0.5, 1, 64


def secondary_c5(dlmz, torch, dev, steps=2, warmup=1):
    """The 7B GQA-shaped workload, a timed prefix: one batch of 64 windows of 2048 tokens, entropy
    threshold 0.5 bits (at least 1, at most 64 positions per step); `warmup` + `steps` denoising
    steps of compression, then the same steps of decompression (which must reproduce the state)."""
    import numpy as np
    from paper_2608_11249_gb300 import sources
    stream = torch.cuda.current_stream().cuda_stream
    V, L, nc = C5["vocab"], C5_CHUNK, C5_BATCH
    m = dlmz.Model(C5["n_layers"], C5["d"], C5["n_heads"], C5["n_kv_heads"], C5["ffn"], V, dlmz.BF16, seed=C5["seed"])
    sym = torch.from_numpy(sources.zipf_bigram_tokens(nc * L, V, seed=0).astype(np.int32).reshape(nc, L)).to(dev)
    state = torch.full((nc, L), V, dtype=torch.int32, device=dev)
    committed = torch.zeros(nc, dtype=torch.int32, device=dev)
    pol = dlmz.policy(dlmz.ENTROPY, 0, 0, C5_TAU, C5_KMIN, C5_KMAX)
    enc = dlmz.Coder(nc, L, V, 24)
    enc.reset_encoder()

    def run(fn):
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        tot = torch.zeros(nc, dtype=torch.int64, device=dev)
        e0, e1 = _events()
        e0.record()
        for _ in range(steps):
            fn()
            tot.add_(committed)  # tokens revealed by this step
        e1.record()
        e1.synchronize()
        return e0.elapsed_time(e1), int(tot.sum().item())

    enc_ms, enc_tok = run(lambda: m.encode_step(enc, pol, 0, L, sym.data_ptr(), state.data_ptr(), committed.data_ptr(),
                                                stream))
    enc_state = state.clone()
    bits = torch.empty(nc, dtype=torch.int32, device=dev)
    cap = enc.capacity_units * 2
    raw = torch.zeros(nc * cap, dtype=torch.uint8, device=dev)
    enc.finish(bits.data_ptr(), raw.data_ptr(), 0, stream)
    offs = (torch.arange(nc, dtype=torch.int64, device=dev) * cap).contiguous()
    dec = dlmz.Coder(nc, L, V, 24)
    dec.load_decoder(raw.data_ptr(), offs.data_ptr(), bits.data_ptr(), stream)
    state.fill_(V)
    dec_ms, dec_tok = run(lambda: m.decode_step(dec, pol, 0, L, state.data_ptr(), committed.data_ptr(), stream))
    dlmz.check(stream)
    assert torch.equal(state, enc_state), "decoder state differs from the encoder's"
    enc.close()
    dec.close()
    m.close()
    del raw, state, enc_state, sym
    torch.cuda.empty_cache()
    return {"workload": "7B GQA-shaped masked DLM, bf16, random-init: 28 layers d=3584 28/4 heads FFN 18944 "
                        "V=152064; 64 windows of 2048 Zipf-bigram tokens, entropy threshold 0.5 bits, at least 1 and "
                        "at most 64 positions per step (a timed prefix of the workload)",
            "compress_Bps": 4.0 * enc_tok / (enc_ms / 1000.0), "decompress_Bps": 4.0 * dec_tok / (dec_ms / 1000.0),
            "ms_per_denoising_step": {"compress": enc_ms / steps, "decompress": dec_ms / steps},
            "tokens_per_step": enc_tok / float(steps), "steps": steps, "warmup": warmup,
            "note": "random-init weights: no position reaches 0.5 bits, so each step reveals m = 1 token per window"}


def secondary_c2(dlmz, torch, dev, steps=2):
    """The byte workload: one 512 KiB batch compressed + decompressed per step (1 warm-up step)."""
    import numpy as np
    from paper_2608_11249_gb300 import sources
    stream = torch.cuda.current_stream().cuda_stream
    m = dlmz.Model(C2["n_layers"], C2["d"], C2["n_heads"], C2["n_kv_heads"], C2["ffn"], C2["vocab"], dlmz.BF16,
                   seed=C2["seed"])
    per = C2_BATCH * C2_CHUNK
    data = sources.markov_bytes(per, seed=0)
    d_in = torch.from_numpy(np.frombuffer(data, dtype=np.uint8).copy()).to(dev)
    cap = m.compress_bound(per, C2_CHUNK)
    d_c = torch.empty(cap, dtype=torch.uint8, device=dev)
    d_out = torch.empty(per, dtype=torch.uint8, device=dev)
    pol = dlmz.policy(dlmz.TOPK_CONF, C2_K, C2_BLOCK)

    def step():
        n = m.compress_device(d_in.data_ptr(), per, C2_CHUNK, pol, d_c.data_ptr(), cap, C2_BATCH, stream)
        m.decompress_device(d_c.data_ptr(), n, d_out.data_ptr(), per, stream)
        return n

    n = step()
    assert torch.equal(d_out, d_in)
    torch.cuda.synchronize()
    e0, e1 = _events()
    e0.record()
    for _ in range(steps):
        n = step()
    e1.record()
    e1.synchronize()
    ms = e0.elapsed_time(e1) / steps
    # one more, untimed step with events around every launch: the kernel split and the rooflines
    prof = dlmz.Profile()
    dlmz.profile_begin()
    step()
    dlmz.profile_end(prof)
    m.close()
    _, _, tf_sus, _ = peaks()
    gi, ai = CLASSES.index("gemm_tcgen05"), CLASSES.index("attention")
    kern_ms = sum(float(prof.ms[j]) for j in range(8))
    split = {c: {"launches": int(prof.n[j]), "ms": round(float(prof.ms[j]), 3), "share": round(float(prof.ms[j]) / kern_ms, 4)}
             for j, c in enumerate(CLASSES) if prof.n[j]}
    frac = lambda j: float(prof.flops[j]) / (float(prof.ms[j]) / 1000.0) / 1e12 / tf_sus if prof.ms[j] else None
    return {"workload": C2_WORKLOAD, "value": per / (ms / 1000.0), "unit": "B/s", "ms_per_step": ms,
            "steps": steps, "warmup": 1, "bits_per_byte": 8.0 * n / per,
            "step": "compress + decompress of one 512 KiB batch (64 + 64 denoising steps), device buffers",
            "kernel_time_split": split,
            "gemm_frac_of_sustained_bf16": frac(gi), "attention_frac_of_sustained_bf16": frac(ai),
            "kernel_split_source": "one more untimed step, CUDA events around every launch"}


def secondary_c3(dlmz, torch, dev, hbm, steps=5):
    """The isolated quantise + select workload at full size (24-bit CDFs + scores, then top-32 of 1024)."""
    R, V, G, K = C3_ROWS, C3_V, C3_GROUP, C3_TOPK
    g = torch.Generator(device=dev).manual_seed(0)
    logits = torch.randn(R, V, device=dev, generator=g)
    logits.mul_(3.0)
    cols = torch.randint(0, V, (R,), device=dev, generator=g)
    logits[torch.arange(R, device=dev), cols] += torch.rand(R, device=dev, generator=g) * 10.0 + 5.0
    cdf = torch.empty(R, V + 1, dtype=torch.int32, device=dev)
    W = torch.empty(R, dtype=torch.int64, device=dev)
    Hq = torch.empty(R, dtype=torch.int32, device=dev)
    keys = torch.empty(R, dtype=torch.int64, device=dev)
    sel = torch.empty(R // G, K, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream().cuda_stream

    def step():
        dlmz.quantize(logits.data_ptr(), R, V, 24, cdf.data_ptr(), W.data_ptr(), 0, Hq.data_ptr(), 0, stream)
        keys.copy_(Hq)
        dlmz.select_smallest(keys.data_ptr(), R // G, G, K, sel.data_ptr(), stream)

    step()
    dlmz.check(stream)
    times = []
    for _ in range(steps):
        e0, e1 = _events()
        e0.record()
        step()
        e1.record()
        e1.synchronize()
        times.append(e0.elapsed_time(e1))
    ms = statistics.median(times)
    alg = R * (4.0 * V + 4.0 * (V + 1))  # logits read + CDF written
    del logits, cdf
    torch.cuda.empty_cache()
    return {"workload": "isolated quantise + select: 65536 x 126464 float32 logits N(0,3) + spike U(5,15), "
                        "24-bit CDFs + W/entropy scores, top-32 of groups of 1024 (inputs > L2)",
            "ms": ms, "rows_per_s": R / (ms / 1000.0), "algorithmic_bytes": alg,
            "achieved_GBps": alg / (ms / 1000.0) / 1e9, "peak_GBps": hbm, "frac": alg / (ms / 1000.0) / 1e9 / hbm,
            "floor_ms": alg / (hbm * 1e9) * 1000.0}


def run(args):
    import torch

    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_11249_gb300 import dlmz

    dev = torch.device("cuda", torch.cuda.current_device())
    hbm, tf_burst, tf_sus, src = peaks()
    r = run_c4(args, dlmz, torch, rank, ws, dev)
    if rank != 0:
        if ws > 1:
            torch.distributed.destroy_process_group()
        return 0
    p = r["prof"]
    gi, ai, qi = CLASSES.index("gemm_tcgen05"), CLASSES.index("attention"), CLASSES.index("quantize")
    kern_ms = sum(p["ms"])
    split = {c: {"launches": p["n"][j], "ms": round(p["ms"][j], 3), "share": round(p["ms"][j] / kern_ms, 4)}
             for j, c in enumerate(CLASSES) if p["n"][j]}
    g_ach = p["flops"][gi] / (p["ms"][gi] / 1000.0) / 1e12 if p["ms"][gi] else 0.0
    a_ach = p["flops"][ai] / (p["ms"][ai] / 1000.0) / 1e12 if p["ms"][ai] else 0.0
    q_ach = p["bytes"][qi] / (p["ms"][qi] / 1000.0) / 1e9 if p["ms"][qi] else 0.0
    secondary = {}
    if not args.no_secondary:
        torch.cuda.empty_cache()
        secondary["byte_workload"] = secondary_c2(dlmz, torch, dev)
        torch.cuda.empty_cache()
        secondary["gqa_7b_prefix"] = secondary_c5(dlmz, torch, dev)
        torch.cuda.empty_cache()
        secondary["quantize_select"] = secondary_c3(dlmz, torch, dev, hbm)
    line = {
        "metric": METRIC, "value": r["value"], "unit": "B/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": r["total_ms"] / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded Zipf(1.05) bigram tokens); random-init N(0,0.02) weights",
        "config": {"workload": C4_WORKLOAD, "batch_chunks": C4_BATCH, "chunk_len": C4_CHUNK, "k": C4_K, "block": 0,
                   "input_bytes_per_step_per_rank": r["step_bytes"],
                   "step": "one denoising step of compression + the matching step of decompression over the batch "
                           "(denoising steps %d..%d of each window timed, %d..%d warm-up)"
                           % (args.warmup, args.warmup + args.steps - 1, 0, args.warmup - 1),
                   "l2": "inputs larger than L2 (weights 16 GB, activations ~48 GB per forward)",
                   "parallelism": "dp%d (independent batches per rank)" % ws},
        "compress_Bps": r["compress_Bps"], "decompress_Bps": r["decompress_Bps"],
        "ms_per_denoising_step": {"compress": r["enc_ms"] / args.steps, "decompress": r["dec_ms"] / args.steps},
        "bits_per_byte": r["bits_per_token_stream"] / 4.0,
        "bits_per_token": r["bits_per_token_stream"],
        "roofline": {"bound": "tensor", "kernel": "tcgen05 GEMM (QKV+RoPE, O+residual, gate/up+SwiGLU, "
                                                  "down+residual, LM head on candidate rows)",
                     "achieved": g_ach, "peak": tf_sus, "unit": "TFLOP/s", "frac": g_ach / tf_sus,
                     "peak_source": "%s bf16_tflops_sustained (kernel timed inside a long step)" % src,
                     "traffic": GEMM_TRAFFIC_PER_LAUNCH,
                     "traffic_source": ("dram__bytes_read.sum + dram__bytes_write.sum of one layer's four GEMM "
                                        "launches at 16 windows (one ncu capture), mean per launch x 32 to 512 "
                                        "windows (traffic grows with the tokens)"),
                     "launches": p["n"][gi],
                     "avg_launch_ms": p["ms"][gi] / p["n"][gi] if p["n"][gi] else None},
        "roofline_attention": {"bound": "tensor", "kernel": "tcgen05 bidirectional attention, head dim 128",
                               "achieved": a_ach, "peak": tf_sus, "unit": "TFLOP/s", "frac": a_ach / tf_sus},
        "roofline_quantize": {"bound": "hbm", "achieved": q_ach, "peak": hbm, "unit": "GB/s", "frac": q_ach / hbm},
        "kernel_time_split": split,
        "gpu_launches": r["launches"],
        "kernel_split_source": ("%d untimed denoising step(s) per direction after the timed ones, CUDA events "
                                "around every launch" % PROF_STEPS),
        "clocks": r["clocks"],
        "e2e": r["e2e"],
        "secondary": secondary,
    }
    if ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(not args.no_cpu_one_thread)
    print(json.dumps(line))
    if ws > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-secondary", action="store_true")
    ap.add_argument("--no-cpu-one-thread", action="store_true", help="time the oracle on all host cores only")
    ap.add_argument("--oracle-child", action="store_true", help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.oracle_child:
        per_step, parts = OracleSampler().sample()
        print(json.dumps({"per_step_s": per_step, "parts": parts}))
        return 0
    if args.impl == "reference":
        return run_reference(args)
    return run(args)


if __name__ == "__main__":
    sys.exit(main())
