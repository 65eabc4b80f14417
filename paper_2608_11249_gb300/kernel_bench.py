"""Runs one piece of the hot path at a chosen size (for ncu captures and timing).

    python -m paper_2608_11249_gb300.kernel_bench forward --chunks 64
        one forward (Definition 3) of the 8-layer d=512 bf16 byte model over
        `chunks` windows of 512 positions (LM head on a 128-row block), repeated --reps times
    python -m paper_2608_11249_gb300.kernel_bench forward --model 8b --layers 2 --chunks 64
        the same for `layers` layers of the 8B-shaped model (d=4096, 32 heads, FFN 12288,
        V=126464) over windows of 1024 positions (LM head on 16 rows per window)
    python -m paper_2608_11249_gb300.kernel_bench quantize --rows 2048 --vocab 126464
        the quantiser (CDF + scores) on spiked N(0,3) logits rows
    python -m paper_2608_11249_gb300.kernel_bench gemm --m 32768 --n 4096 --k 512
        one bf16 tensor-core GEMM with float32 output
    python -m paper_2608_11249_gb300.kernel_bench step --layers 1 --chunks 16 [--decode]
        one denoising step of compression (forward, LM head and quantiser on the
        candidates, selection, range coding of 16 tokens per window) of the
        8B-shaped model with `layers` layers over `chunks` windows of 1024 tokens;
        --decode: one step is compressed untimed, then its decompression is timed

Prints the mean CUDA-event time per repetition.
"""
import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    import numpy as np
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_11249_gb300 import dlmz

    ap = argparse.ArgumentParser()
    ap.add_argument("what", choices=["forward", "quantize", "gemm", "step"])
    ap.add_argument("--chunks", type=int, default=64)
    ap.add_argument("--rows", type=int, default=2048)
    ap.add_argument("--vocab", type=int, default=126464)
    ap.add_argument("--m", type=int, default=32768)
    ap.add_argument("--n", type=int, default=4096)
    ap.add_argument("--k", type=int, default=512)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--model", choices=["byte", "8b"], default="byte")
    ap.add_argument("--layers", type=int, default=2)
    ap.add_argument("--decode", action="store_true")
    a = ap.parse_args()
    torch.cuda.set_device(0)
    g = torch.Generator(device="cuda").manual_seed(0)
    if a.what == "step":
        from paper_2608_11249_gb300 import sources
        V, L, k = 126464, 1024, 16
        m = dlmz.Model(a.layers, 4096, 32, 32, 12288, V, dlmz.BF16, seed=0)
        m.set_logits_budget(2 << 30)  # candidate logits in slabs of 2 GiB (small device footprint)
        sym = torch.from_numpy(sources.zipf_bigram_tokens(a.chunks * L, V, seed=0).astype(np.int32)).cuda()
        state = torch.full((a.chunks, L), V, dtype=torch.int32, device="cuda")
        enc = dlmz.Coder(a.chunks, L, V, 24)
        enc.reset_encoder()
        pol = dlmz.policy(dlmz.TOPK_CONF, k, 0)
        a.reps = min(a.reps, L // k - 1)
        fn = lambda: m.encode_step(enc, pol, 0, L, sym.data_ptr(), state.data_ptr())
        if a.decode:  # compress 1 + reps steps, then time their decompression (1 untimed + reps)
            for _ in range(1 + a.reps):
                fn()
            bits = torch.empty(a.chunks, dtype=torch.int32, device="cuda")
            cap = enc.capacity_units * 2
            raw = torch.zeros(a.chunks * cap, dtype=torch.uint8, device="cuda")
            enc.finish(bits.data_ptr(), raw.data_ptr())
            offs = torch.arange(a.chunks, dtype=torch.int64, device="cuda") * cap
            dec = dlmz.Coder(a.chunks, L, V, 24)
            dec.load_decoder(raw.data_ptr(), offs.data_ptr(), bits.data_ptr())
            state.fill_(V)
            fn = lambda: m.decode_step(dec, pol, 0, L, state.data_ptr())
    elif a.what == "forward" and a.model == "8b":
        V, L, rpc = 126464, 1024, 16
        m = dlmz.Model(a.layers, 4096, 32, 32, 12288, V, dlmz.BF16, seed=0)
        state = torch.randint(0, V + 1, (a.chunks, L), dtype=torch.int32, device="cuda", generator=g)
        logits = torch.empty(a.chunks * rpc, V, dtype=torch.float32, device="cuda")
        fn = lambda: m.forward_logits(state.data_ptr(), a.chunks, L, 0, rpc, logits.data_ptr())
    elif a.what == "forward":
        m = dlmz.Model(8, 512, 8, 8, 2048, 256, dlmz.BF16, seed=0)
        L = 512
        state = torch.randint(0, 257, (a.chunks, L), dtype=torch.int32, device="cuda", generator=g)
        logits = torch.empty(a.chunks * 128, 256, dtype=torch.float32, device="cuda")
        fn = lambda: m.forward_logits(state.data_ptr(), a.chunks, L, 128, 128, logits.data_ptr())
    elif a.what == "quantize":
        V = a.vocab
        x = torch.randn(a.rows, V, device="cuda", generator=g) * 3
        x[torch.arange(a.rows), torch.randint(0, V, (a.rows,), device="cuda", generator=g)] += 10
        cdf = torch.empty(a.rows, V + 1, dtype=torch.int32, device="cuda")
        W = torch.empty(a.rows, dtype=torch.int64, device="cuda")
        Hq = torch.empty(a.rows, dtype=torch.int32, device="cuda")
        P = 16 if V <= 4096 else 24
        fn = lambda: dlmz.quantize(x.data_ptr(), a.rows, V, P, cdf.data_ptr(), W.data_ptr(), 0, Hq.data_ptr(), 0)
    else:
        A = (torch.randn(a.m, a.k, device="cuda", generator=g)).to(torch.bfloat16)
        B = (torch.randn(a.n, a.k, device="cuda", generator=g)).to(torch.bfloat16)
        D = torch.empty(a.m, a.n, dtype=torch.float32, device="cuda")
        fn = lambda: dlmz.gemm_bf16(A.data_ptr(), B.data_ptr(), D.data_ptr(), a.m, a.n, a.k)
    fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(a.reps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    dlmz.check()
    ms = e0.elapsed_time(e1) / a.reps
    extra = ""
    if a.what == "gemm":
        extra = " %.1f TFLOP/s" % (2.0 * a.m * a.n * a.k / ms / 1e9)
    elif a.what == "quantize":
        extra = " %.1f GB/s (logits read + CDF write)" % ((4.0 * a.rows * a.vocab * 2) / ms / 1e6)
    print("%s: %.3f ms per repetition%s" % (a.what, ms, extra))


if __name__ == "__main__":
    main()
