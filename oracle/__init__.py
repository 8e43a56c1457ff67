"""Float64 CPU oracle for the cross-model KV-cache mapper (arXiv 2608.03893).

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only ``tests/``, ``__graft_entry__.smoke()``
and the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import or run
anything in this package.  The product path (the ``kvx`` C-ABI library and its Python
binding) never calls it, and this package never imports the product.

Everything here is a plain, slow, obviously-correct restatement of what the paper
defines, in float64 numpy, one function per defined quantity:

* ``rope``      -- the RoPE rotation R_Theta(t) and its inverse (Sec. 3.3).
* ``bf16``      -- exact bf16 decoding and round-to-nearest-even encoding, used to
                   express the bf16 forward of Appendix "Run information".
* ``selection`` -- top-k source-layer selection per target layer (Sec. 3.2).
* ``r2``        -- the single-source OLS probe and its head-averaged R^2
                   (Sec. 2.3, Eq. single_source_ols) and the selection score.
* ``ridge``     -- the centred closed-form ridge fit (Sec. 3.1, Eq. Wstar).
* ``mapper``    -- applying the fitted mapper: strip source RoPE, concatenate the
                   k selected layers, X W + b, re-apply target RoPE (Eq. ridge_kv,
                   Sec. 3.2 concatenation, Sec. 3.3 content-space composition);
                   plus the mapper-size formula of Appendix C.
* ``mlp``       -- applying the MLP mapper of Sec. 4.3 / Appendix "Run information"
                   (three Linear layers with ReLU on the cross-head source feature).

Pins (tests/test_oracle_*.py, run with ``-m "not gpu"``) tie each function to
something other than itself: closed forms, textbook routines, brute force and the
paper's printed mapper-size table.  The paper prints no worked numeric example of a
mapping, so the mapping itself is pinned by invariants and brute force only.
"""
