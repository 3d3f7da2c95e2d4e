"""CPU oracle for the TASP compiled sparse execution path.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import, call, link or execute anything in
this package. The product (the CUDA library and its Python binding) never
touches it, and it shares no code with the product: it has its own quantizer,
FLOP ledger, mask compiler, panel packer and forward pass, written from the
paper, plus its own C regenerator of the synthetic weights. The only common
module is ``synth`` (seeded input generation, no arithmetic of the method).

Definition of the forward (the paper's "mask-as-zero" control, Table 3, and
the exactness of structured removal): for a mask M the dense dequantized FP32
weights W~ = s * Q are formed per output row, the pruned units are ZEROED
(Q/K/V rows of dropped GQA groups, O-projection columns of their query heads,
gate/up rows and down columns of dropped SwiGLU channels; Sec. 3.3), and the
plain Llama decoder runs in FP32. Compacted execution is an exact
reformulation of this because zero rows/columns contribute exactly zero.

Parity status of each function is listed in its module header.
"""
