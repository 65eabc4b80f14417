"""Writes the golden fixtures of this folder from the oracle alone.

Run from the repository root:  python tests/golden/make_golden.py
Every value stored here comes from ``oracle/`` (the paper prints no worked
example); the fixtures freeze the oracle's definitions so that a change to
its arithmetic shows up as a failing test.
"""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import coder, model, quantizer, selector, pipeline  # noqa: E402


def main():
    g = {}
    # Quantiser table T and constant C (integer CDF rule).
    g["exp_table"] = [int(t) for t in quantizer.exp_table()]
    g["scale_constant_bits"] = int(np.float32(quantizer.scale_constant()).view(np.uint32))
    # One 8-symbol row through the quantiser (P = 16).
    row = np.array([[0.5, -1.25, 3.0, 3.0, 0.0, -7.5, 2.25, 1.0]], dtype=np.float32)
    q = quantizer.quantize(row, 16)
    g["quantize_row"] = {"logits": row[0].tolist(), "cdf": q["cdf"][0].tolist(), "W": int(q["W"][0]),
                         "Hq": int(q["Hq"][0]), "top": int(q["top"][0])}
    # Range coder: fixed (c, f) pairs at P = 16.
    pairs = [(0, 1), (65535, 1), (100, 30000), (40000, 25536), (1, 2), (32768, 32768)] * 7
    enc = coder.Encoder(16)
    for c, f in pairs:
        enc.encode(c, f)
    bits, data = enc.finish()
    g["range_coder"] = {"P": 16, "pairs": pairs, "bits": bits, "hex": data.hex()}
    # Tiny f32 model: logits of one state, and a full container.
    cfg = model.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=1, ffn=16, vocab=4, dtype="f32", seed=1)
    w = model.Weights(cfg)
    state = [4, 0, 3, 4, 1]
    g["tiny_model_logits"] = {"state": state, "logits": model.forward(w, np.array(state)).tolist()}
    pol = selector.Policy(kind=selector.TOPK_CONF, k=2, block=4)
    data_in = bytes([0, 1, 2, 3, 3, 2, 1, 0, 1, 1, 2])
    blob = pipeline.compress(w, data_in, 8, pol)
    g["tiny_container"] = {"input_hex": data_in.hex(), "chunk_len": 8, "k": 2, "block": 4, "hex": blob.hex()}
    with open(os.path.join(HERE, "oracle_fixtures.json"), "w") as fh:
        json.dump(g, fh, indent=1)
        fh.write("\n")


if __name__ == "__main__":
    main()
