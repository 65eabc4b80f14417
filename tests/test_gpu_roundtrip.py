"""End-to-end GPU compress / decompress through the C ABI.

Round trips must be bit-exact; the GPU container's size must be within
0.5% of the oracle's own end-to-end compression of the same input with the
same model (the two forwards differ by rounding, so the streams differ).
"""
import numpy as np
import pytest

from oracle import container as OC
from oracle import context as OX
from oracle import model as OM
from oracle import pipeline as OP
from oracle import selector as S
from paper_2608_11249_gb300 import sources
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = pytest.mark.gpu

CASES = [
    # model (nl, d, h, kv, F, V, dtype), data kind, n, chunk_len, policy, batch_chunks
    ((1, 32, 2, 2, 64, 256, "f32"), "bytes", 1500, 512, S.Policy(kind=S.TOPK_CONF, k=4, block=64), 0),
    ((2, 256, 4, 4, 256, 256, "bf16"), "bytes", 1100, 256, S.Policy(kind=S.TOPK_CONF, k=8, block=128), 3),
    ((1, 64, 4, 2, 128, 5000, "f32"), "tokens", 300, 100, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=8), 0),
    ((2, 256, 4, 4, 256, 256, "bf16"), "bytes", 600, 200, S.Policy(kind=S.ENTROPY, tau_bits=6.0, k_min=2, k_max=16), 2),
]


def _data(kind, n, V):
    if kind == "bytes":
        return sources.markov_bytes(n, seed=2)
    return sources.tokens_to_bytes(sources.zipf_bigram_tokens(n, V, seed=2))


def _model(d, spec, seed):
    nl, dm, h, kv, F, V, dt = spec
    return d.Model(nl, dm, h, kv, F, V, d.BF16 if dt == "bf16" else d.FP32, seed=seed)


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_roundtrip_and_size_vs_oracle(dev, ci):
    d = dlmz()
    spec, kind, n, L, opol, bc = CASES[ci]
    m = _model(d, spec, 40 + ci)
    data = _data(kind, n, spec[5])
    pol = d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max)
    blob = m.compress(data, L, pol, bc)
    assert m.decompress(blob) == data
    h, streams = OC.read(blob)  # the oracle's container reader parses the GPU file
    assert h.fingerprint == m.fingerprint and h.chunk_len == L and h.n_symbols * (4 if kind == "tokens" else 1) == len(data)
    w = OM.Weights(OM.ModelConfig(*spec, seed=40 + ci))
    oblob = OP.compress(w, data, L, opol)
    assert abs(len(blob) - len(oblob)) <= 0.005 * len(oblob) + 8, (len(blob), len(oblob))


LR_CASES = [
    # model, data kind, n, chunk_len, oracle policy, context (kind, c, seed), batch_chunks
    ((1, 32, 2, 2, 64, 256, "f32"), "bytes", 1500, 512, S.Policy(kind=S.UNIFORM, k=16), (OX.NONE, 0, 0), 0),
    ((2, 256, 4, 4, 256, 256, "bf16"), "bytes", 1100, 256, S.Policy(kind=S.PROGRESSIVE, k=2, growth_q16=98304),
     (OX.RANDOM, 8, 5), 3),
    ((1, 64, 4, 2, 128, 5000, "f32"), "tokens", 300, 100, S.Policy(kind=S.UNIFORM, k=7), (OX.CONTIGUOUS, 5, 0), 0),
    ((2, 256, 4, 4, 256, 256, "bf16"), "bytes", 600, 200, S.Policy(kind=S.TOPK_CONF, k=8, block=64),
     (OX.RANDOM, 16, 9), 2),
    ((2, 256, 4, 4, 256, 256, "bf16"), "bytes", 600, 200, S.Policy(kind=S.ENTROPY, tau_bits=6.0, k_min=2, k_max=16),
     (OX.CONTIGUOUS, 3, 0), 2),
    ((1, 32, 2, 2, 64, 256, "f32"), "bytes", 700, 64, S.Policy(kind=S.PROGRESSIVE, k=1, growth_q16=2 << 16),
     (OX.RANDOM, 100, 3), 0),  # c > window: whole windows stored as context
]


@pytest.mark.parametrize("ci", range(len(LR_CASES)))
def test_schedules_and_context_vs_oracle(dev, ci):
    """Uniform/progressive schedules (Sec. 3.3) and initial context (Sec. 3.4): round trip, the stored
    context symbols bit for bit, and the container size against the oracle's own compression."""
    d = dlmz()
    spec, kind, n, L, opol, ctx, bc = LR_CASES[ci]
    m = _model(d, spec, 60 + ci)
    data = _data(kind, n, spec[5])
    pol = d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max, opol.growth_q16,
                   ctx[0], ctx[1], ctx[2])
    blob = m.compress(data, L, pol, bc)
    assert m.decompress(blob) == data
    h, streams = OC.read(blob)
    assert (h.ctx_kind, h.ctx_c, h.ctx_seed) == (ctx if ctx[1] else (0, 0, 0))
    sym = np.frombuffer(data, dtype=np.uint8 if kind == "bytes" else "<u4").astype(np.int64)
    want = []
    for c in range(h.n_chunks):
        win = sym[c * L:(c + 1) * L]
        want.append(win[OX.positions(ctx[0], ctx[1], ctx[2], win.size, c)])
    want = np.concatenate(want) if want else np.zeros(0, dtype=np.int64)
    assert h.ctx_data == (want.astype(np.uint8).tobytes() if kind == "bytes" else want.astype("<u4").tobytes())
    w = OM.Weights(OM.ModelConfig(*spec, seed=60 + ci))
    oblob = OP.compress(w, data, L, opol, context=ctx)
    assert abs(len(blob) - len(oblob)) <= 0.005 * len(oblob) + 8, (len(blob), len(oblob))


RANS_RT = [
    ((1, 32, 2, 2, 64, 256, "f32"), "bytes", 1500, 512, S.Policy(kind=S.TOPK_CONF, k=4, block=64), (OX.NONE, 0, 0), 0),
    ((2, 256, 4, 4, 256, 256, "bf16"), "bytes", 1100, 256, S.Policy(kind=S.UNIFORM, k=32), (OX.RANDOM, 8, 5), 3),
    ((1, 64, 4, 2, 128, 5000, "f32"), "tokens", 300, 100, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=8),
     (OX.NONE, 0, 0), 0),
]


@pytest.mark.parametrize("ci", range(len(RANS_RT)))
def test_rans_roundtrip_and_size_vs_oracle(dev, ci):
    """Whole files with the rANS coder: round trip, header coder byte, size against the oracle's rANS file."""
    d = dlmz()
    spec, kind, n, L, opol, ctx, bc = RANS_RT[ci]
    m = _model(d, spec, 80 + ci)
    data = _data(kind, n, spec[5])
    pol = d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max, opol.growth_q16,
                   ctx[0], ctx[1], ctx[2], coder=d.CODER_RANS)
    blob = m.compress(data, L, pol, bc)
    assert m.decompress(blob) == data
    h, streams = OC.read(blob)
    assert h.coder == 1 and all(b % 32 == 0 and b >= 64 for b, _ in streams)
    w = OM.Weights(OM.ModelConfig(*spec, seed=80 + ci))
    oblob = OP.compress(w, data, L, opol, context=ctx, coder=OP.RANS)
    assert abs(len(blob) - len(oblob)) <= 0.005 * len(oblob) + 8, (len(blob), len(oblob))
    rblob = m.compress(data, L, d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max,
                                         opol.growth_q16, ctx[0], ctx[1], ctx[2]), bc)
    assert len(blob) - len(rblob) <= 13 * h.n_chunks + 8  # rANS: at most ~96 bits more per window than the range coder


def test_ranks_roundtrip_and_size_vs_oracle(dev):
    """Whole files with symbol ranks: round trip, coder byte, size against the oracle's rank file."""
    d = dlmz()
    spec = (1, 32, 2, 2, 64, 256, "f32")
    m = _model(d, spec, 90)
    data = _data("bytes", 1200, 256)
    opol = S.Policy(kind=S.TOPK_CONF, k=4, block=64)
    pol = d.policy(opol.kind, opol.k, opol.block, coder=d.CODER_RANKS)
    blob = m.compress(data, 256, pol)
    assert m.decompress(blob) == data
    h, streams = OC.read(blob)
    assert h.coder == 2 and all(b % 8 == 0 for b, _ in streams)
    w = OM.Weights(OM.ModelConfig(*spec, seed=90))
    oblob = OP.compress(w, data, 256, opol, coder=OP.RANKS)
    assert abs(len(blob) - len(oblob)) <= 0.005 * len(oblob) + 8, (len(blob), len(oblob))
    for i in (80, len(blob) // 2, len(blob) - 1):  # edited rank bytes: rejected, never a crash
        bad = blob[:i] + bytes([blob[i] ^ 0x40]) + blob[i + 1:]
        try:
            out = m.decompress(bad)
        except d.DlmzError as e:
            assert e.code == d.ECORRUPT
        else:
            assert out == data
    d.check()


def test_bad_schedule_and_context_rejected(dev):
    d = dlmz()
    m = _model(d, (1, 32, 2, 2, 64, 256, "f32"), 1)
    for pol in (d.policy(d.UNIFORM, 0), d.policy(d.PROGRESSIVE, 1, growth_q16=0),
                d.policy(d.PROGRESSIVE, 1, growth_q16=(64 << 16) + 1), d.policy(d.TOPK_CONF, 2, context=d.CONTEXT_RANDOM),
                d.policy(d.TOPK_CONF, 2, context=7, context_c=1), d.policy(d.TOPK_CONF, 2, context_c=3),
                d.policy(d.TOPK_CONF, 2, coder=3)):
        with pytest.raises(d.DlmzError) as e:
            m.compress(b"abcdef", 4, pol)
        assert e.value.code == d.EINVAL
    blob = m.compress(b"abcdefgh", 4, d.policy(d.UNIFORM, 2, context=d.CONTEXT_RANDOM, context_c=2, context_seed=1))
    # bad context kind, truncated extension, an edited context symbol (the checksum catches it)
    for bad in (blob[:64] + b"\x09" + blob[65:], blob[:79], blob[:80] + bytes([blob[80] ^ 1]) + blob[81:]):
        with pytest.raises(d.DlmzError) as e:
            m.decompress(bad)
        assert e.value.code == d.ECORRUPT
    d.check()


def test_edge_inputs(dev):
    d = dlmz()
    m = _model(d, (1, 32, 2, 2, 64, 256, "f32"), 1)
    pol = d.policy(d.TOPK_CONF, 3, 8)
    for data in (b"", b"\x07", bytes(range(256)), b"\xff" * 33):
        blob = m.compress(data, 16, pol)
        assert m.decompress(blob) == data
    tm = _model(d, (1, 32, 2, 2, 64, 300, "f32"), 1)
    with pytest.raises(d.DlmzError) as e:
        tm.compress(b"\x01\x02\x03", 16, pol)
    assert e.value.code == d.EBADINPUT
    with pytest.raises(d.DlmzError) as e:
        tm.compress(np.array([300], dtype="<u4").tobytes(), 16, pol)
    assert e.value.code == d.EBADINPUT
    with pytest.raises(d.DlmzError):
        m.compress(b"abc", 0, pol)
    with pytest.raises(d.DlmzError):
        m.compress(b"abc", 4, d.policy(d.TOPK_CONF, 0))


def test_device_api_matches_host_api_and_batches_agree(dev):
    import torch
    d = dlmz()
    m = _model(d, (2, 256, 4, 4, 256, 256, "bf16"), 7)
    data = sources.markov_bytes(2000, seed=5)
    pol = d.policy(d.TOPK_CONF, 8, 64)
    a = m.compress(data, 256, pol, 1)
    b = m.compress(data, 256, pol, 4)
    # batch composition changes no stream (batch-invariant forward): only the header's batch field differs
    assert a[:24] == b[:24] and a[28:] == b[28:]
    din = to_dev(np.frombuffer(data, dtype=np.uint8))
    cap = m.compress_bound(len(data), 256)
    dout = torch.empty(cap, dtype=torch.uint8, device="cuda")
    n = m.compress_device(ptr(din), len(data), 256, pol, ptr(dout), cap, batch_chunks=4)
    assert bytes(dout[:n].cpu().numpy()) == b
    back = torch.empty(len(data), dtype=torch.uint8, device="cuda")
    k = m.decompress_device(ptr(dout), n, ptr(back), len(data))
    assert k == len(data) and bytes(back.cpu().numpy()) == data


def test_corrupt_containers_are_rejected(dev):
    d = dlmz()
    m = _model(d, (1, 32, 2, 2, 64, 256, "f32"), 9)
    data = sources.markov_bytes(400, seed=9)
    blob = m.compress(data, 128, d.policy(d.TOPK_CONF, 4, 32))
    bad = [b"XXXX" + blob[4:], blob[:4] + b"\x09" + blob[5:], blob[:-1], blob[:30], blob + b"\0"]
    for x in bad:
        with pytest.raises(d.DlmzError) as e:
            m.decompress(x)
        assert e.value.code == d.ECORRUPT
    other = _model(d, (1, 32, 2, 2, 64, 256, "f32"), 10)
    with pytest.raises(d.DlmzError) as e:
        other.decompress(blob)
    assert e.value.code == d.EMODEL
    rng = np.random.default_rng(0)
    for _ in range(20):  # flipped bits: rejected by the checksum or the coder, never a crash;
        x = bytearray(blob)  # a flip inside a stream's final zero padding may still decode correctly
        i = int(rng.integers(70, len(x)))
        x[i] ^= 1 << int(rng.integers(0, 8))
        try:
            out = m.decompress(bytes(x))
        except d.DlmzError as e:
            assert e.code == d.ECORRUPT
        else:
            assert out == data
    d.check()


SLAB_CASES = [
    # model, data kind, n, chunk_len, policy (kind, k, block, tau, k_min, k_max), context, batch_chunks
    ((1, 64, 4, 2, 128, 5000, "f32"), "tokens", 700, 100, (S.TOPK_CONF, 8, 0, 0.0, 1, 0), (OX.NONE, 0, 0), 3),
    ((2, 256, 4, 4, 256, 5000, "bf16"), "tokens", 500, 128, (S.ENTROPY, 0, 0, 0.5, 1, 8), (OX.RANDOM, 9, 2), 2),
    ((1, 64, 4, 2, 128, 5000, "f32"), "tokens", 400, 100, (S.UNIFORM, 6, 0, 0.0, 1, 0), (OX.NONE, 0, 0), 0),
    ((1, 32, 2, 2, 64, 256, "f32"), "bytes", 900, 300, (S.TOPK_CONF, 4, 64, 0.0, 1, 0), (OX.RANDOM, 20, 7), 2),
]


@pytest.mark.parametrize("ci", range(len(SLAB_CASES)))
def test_candidate_slabs_give_identical_files(dev, ci):
    """The LM head and quantiser run on the candidate rows; with a logits budget of a few
    rows they run in slabs and the selected rows are recomputed for the coder.  The file
    must not depend on the budget, and either model decodes it."""
    d = dlmz()
    spec, kind, n, L, (k0, k, blk, tau, kmin, kmax), ctx, bc = SLAB_CASES[ci]
    data = _data(kind, n, spec[5])
    pol = d.policy(k0, k, blk, tau, kmin, kmax, 65536, ctx[0], ctx[1], ctx[2])
    a = _model(d, spec, 120 + ci)
    blob = a.compress(data, L, pol, bc)
    b = _model(d, spec, 120 + ci)
    b.set_logits_budget(7 * spec[5] * 4)  # 7 rows of logits: many slabs per step
    assert b.compress(data, L, pol, bc) == blob
    assert b.decompress(blob) == data
    assert a.decompress(blob) == data


@pytest.mark.parametrize("spec,V,L,nc,pol_args", [
    ((2, 256, 4, 4, 256, 256, "bf16"), 256, 128, 4, (S.TOPK_CONF, 8, 64, 0.0, 1, 0)),
    ((1, 64, 4, 2, 128, 5000, "f32"), 5000, 96, 3, (S.ENTROPY, 0, 0, 0.5, 1, 8)),
])
def test_model_step_api_matches_whole_file(dev, spec, V, L, nc, pol_args):
    """dlmz_model_encode_step / dlmz_model_decode_step over one batch: the streams equal those of
    the dlmz_compress file of the same windows, and decoding recovers the symbols."""
    import torch
    from oracle import quantizer as Q
    d = dlmz()
    m = _model(d, spec, 150)
    kind = "bytes" if V == 256 else "tokens"
    data = _data(kind, nc * L, V)
    sym = np.frombuffer(data, dtype=np.uint8 if kind == "bytes" else "<u4").astype(np.int32).reshape(nc, L)
    k0, k, blk, tau, kmin, kmax = pol_args
    pol = d.policy(k0, k, blk, tau, kmin, kmax)
    blob = m.compress(data, L, pol, nc)
    _, want = OC.read(blob)
    P = Q.precision_for_vocab(V)
    coder = d.Coder(nc, L, V, P)
    coder.reset_encoder()
    d_sym = to_dev(sym)
    state = to_dev(np.full((nc, L), V, dtype=np.int32))
    committed = torch.zeros(nc, dtype=torch.int32, device="cuda")
    B = blk or L

    def run(step_fn):
        if k0 == S.TOPK_CONF:
            for b0 in range(0, L, B):
                for _ in range(-(-min(B, L - b0) // k)):
                    step_fn(b0, min(B, L - b0))
        else:
            for _ in range(L + 1):
                if int((state == V).sum().item()) == 0:
                    break
                step_fn(0, L)

    run(lambda r0, rpc: m.encode_step(coder, pol, r0, rpc, ptr(d_sym), ptr(state), ptr(committed)))
    d.check()
    assert np.array_equal(state.cpu().numpy(), sym)
    bits = torch.empty(nc, dtype=torch.int32, device="cuda")
    cap = coder.capacity_units * 2
    raw = torch.zeros(nc * cap, dtype=torch.uint8, device="cuda")
    coder.finish(ptr(bits), ptr(raw))
    d.check()
    bits_h = bits.cpu().numpy().astype(np.int64)
    raw_h = raw.cpu().numpy()
    got = [(int(bits_h[c]), bytes(raw_h[c * cap:c * cap + (bits_h[c] + 7) // 8])) for c in range(nc)]
    assert got == [(int(b), bytes(s)) for b, s in want]
    packed = np.frombuffer(b"".join(s for _, s in got) + b"\0" * 8, dtype=np.uint8)
    offs = np.concatenate([[0], np.cumsum([(b + 7) // 8 for b in bits_h])[:-1]]).astype(np.int64)
    dec = d.Coder(nc, L, V, P)
    d_packed, d_offs, d_bits = to_dev(packed), to_dev(offs), to_dev(bits_h.astype(np.int32))
    dec.load_decoder(ptr(d_packed), ptr(d_offs), ptr(d_bits))
    state.copy_(to_dev(np.full((nc, L), V, dtype=np.int32)))
    run(lambda r0, rpc: m.decode_step(dec, pol, r0, rpc, ptr(state), ptr(committed)))
    d.check()
    assert np.array_equal(state.cpu().numpy(), sym)


def test_model_step_matches_logits_step_large_vocabulary(dev):
    """V > 512: the model-driven step quantises its candidates from the LM head epilogue's row
    maxima (one read of each logit); the logits-driven step reads the same logits twice.  Both
    must give the same streams."""
    import torch
    d = dlmz()
    V, L, nc, k, blk = 1024, 128, 3, 8, 64
    m = d.Model(1, 256, 4, 4, 256, V, d.BF16, seed=77)
    sym = to_dev(np.random.default_rng(5).integers(0, V, (nc, L)).astype(np.int32))
    pol = d.policy(S.TOPK_CONF, k, blk)
    streams = []
    from oracle import quantizer as Q
    for driven_by_model in (True, False):
        coder = d.Coder(nc, L, V, Q.precision_for_vocab(V))
        coder.reset_encoder()
        state = to_dev(np.full((nc, L), V, dtype=np.int32))
        logits = torch.empty(nc * blk, V, dtype=torch.float32, device="cuda")
        for b0 in range(0, L, blk):
            for _ in range(blk // k):
                if driven_by_model:
                    m.encode_step(coder, pol, b0, blk, ptr(sym), ptr(state))
                else:
                    m.forward_logits(ptr(state), nc, L, b0, blk, ptr(logits))
                    coder.encode_step(pol, ptr(logits), b0, blk, ptr(sym), ptr(state))
        d.check()
        assert torch.equal(state, sym)
        bits = torch.empty(nc, dtype=torch.int32, device="cuda")
        raw = torch.zeros(nc * coder.capacity_units * 2, dtype=torch.uint8, device="cuda")
        coder.finish(ptr(bits), ptr(raw))
        d.check()
        streams.append((bits.cpu().numpy().copy(), raw.cpu().numpy().copy()))
        coder.close()
    assert np.array_equal(streams[0][0], streams[1][0])
    assert np.array_equal(streams[0][1], streams[1][1])
    m.close()
