"""Slow, plain CPU oracle for the DLM compression hot path.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports this package:
only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may use it.  It shares no code,
tables or constants generators with the CUDA library under
``paper_2608_11249_gb300/``; the two meet only through the seeded input
generators in ``paper_2608_11249_gb300/sources.py`` (which hold none of the
method's arithmetic).

Modules, each following the paper ("Diffuse to Compress: Leveraging
Diffusion LMs for Lossless Compression"):

* ``weights``   -- counter-based N(0, 0.02) initialisation (SplitMix64 +
                   Box-Muller) standing in for trained weights.
* ``model``     -- the masked, bidirectional diffusion-LM forward pass of
                   Definition 3 (Sec. 3.1), float64 with the storage
                   rounding of the model's dtype.
* ``quantizer`` -- logits -> integer frequencies / CDF + confidence and
                   entropy scores (Sec. 3.3 entropy equation; rANS-style
                   statistical coding of Sec. 2.1 / Sec. 4).
* ``selector``  -- commitment schedules of Sec. 3.3 (max-confidence top-k in
                   left-to-right blocks, entropy threshold with minimum m,
                   uniform block, progressive).
* ``context``   -- initial context of Sec. 3.4 (contiguous, random).
* ``coder``     -- range coder with minimal termination (statistical coding,
                   Sec. 2.1 and Sec. 4 "Implementation Details").
* ``rans``      -- rANS coder (64-bit state, 32-bit words), the paper's coder.
* ``ranking``   -- symbol ranking with varint output (the paper's ranking pipeline).
* ``container`` -- compressed-file header (Sec. 3.3 last paragraph, Sec. 4).
* ``pipeline``  -- the iterative pipeline S^(k+1) = f_theta(S^(k)) of
                   Sec. 3.2, compress and decompress.

Parity status per function is recorded in each module's docstring.
"""
