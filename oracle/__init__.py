"""CPU oracle for the W8A8 SmoothQuant hot path (test infrastructure, not product code).

This package is a plain, slow, step-by-step restatement of what the paper defines:
the SmoothQuant smoothing factor (Eq. delta-attn / delta-lmhead), the smoothed operands
(Eq. xhat-lmhead, what-lmhead), per-output-channel weight quantisation (Eq. si, what-ffn),
dynamic per-token activation quantisation (Eq. stx, xint8), the INT8 GEMM with its
dequantising scale (Eq. gemm-final), the layer-group masks (Eq. ffn55, ffn1010, ffnall26,
attnffn55, attnffn1010), the quality metrics (Top-1 agreement and perplexity delta of the
LM Head section, SQNR of Eq. sqnr-ffn / sqnr-block) and the allocation rule of the
Problem Statement and Combined Configurations sections.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s ``cpu_baseline`` /
``--impl reference`` legs may import, call or execute anything in this package.  The
product path (the CUDA library and its Python binding) never imports it, and this package
never imports the product path: the two share no code.  Inputs reach both sides from the
seeded generators in ``synth/``, which hold none of the method's arithmetic.

Parity status per module (what pins each function is listed in its docstring):
  w8a8.py      pinned: brute force in exact integer/rational arithmetic, invariants,
               the textbook special case (delta = 1, integer grid, s = 1).
  geglu.py     pinned: closed forms of tanh/GELU, fp64 definition within a stated bound.
  masks.py     pinned: set equality with the paper's equations; Table 1 weight sizes.
  quality.py   pinned: the paper's printed ratios (179/181, 10.0495/9.9652).
  allocator.py pinned: the paper's combined-configuration table and its stated choice.
  decoder.py   parity unpinned: the paper gives no numbers for a random-init decoder;
               only its parts (RMSNorm, RoPE, softmax attention) are pinned by textbook
               identities in the tests.
"""
