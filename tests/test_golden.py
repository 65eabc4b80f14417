"""The oracle reproduces its frozen golden fixtures (tests/golden/)."""
import json
import os

import numpy as np

from oracle import coder, model, pipeline, quantizer, selector

G = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "oracle_fixtures.json")))


def test_tables():
    assert [int(t) for t in quantizer.exp_table()] == G["exp_table"]
    assert int(np.float32(quantizer.scale_constant()).view(np.uint32)) == G["scale_constant_bits"]


def test_quantize_row():
    g = G["quantize_row"]
    q = quantizer.quantize(np.array([g["logits"]], dtype=np.float32), 16)
    assert q["cdf"][0].tolist() == g["cdf"] and int(q["W"][0]) == g["W"]
    assert int(q["Hq"][0]) == g["Hq"] and int(q["top"][0]) == g["top"]


def test_range_coder_stream():
    g = G["range_coder"]
    enc = coder.Encoder(g["P"])
    for c, f in g["pairs"]:
        enc.encode(c, f)
    bits, data = enc.finish()
    assert bits == g["bits"] and data.hex() == g["hex"]


def test_tiny_model_and_container():
    cfg = model.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=1, ffn=16, vocab=4, dtype="f32", seed=1)
    w = model.Weights(cfg)
    g = G["tiny_model_logits"]
    assert np.allclose(model.forward(w, np.array(g["state"])), np.array(g["logits"]), atol=1e-7)
    g = G["tiny_container"]
    pol = selector.Policy(kind=selector.TOPK_CONF, k=g["k"], block=g["block"])
    blob = pipeline.compress(w, bytes.fromhex(g["input_hex"]), g["chunk_len"], pol)
    assert blob.hex() == g["hex"]
    assert pipeline.decompress(w, blob) == bytes.fromhex(g["input_hex"])
