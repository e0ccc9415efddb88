"""CPU oracle for the AtSpeed verification call (arXiv 2410.05165).

TEST INFRASTRUCTURE ONLY.  Plain, slow, obviously-correct NumPy code that the
parity tests, ``__graft_entry__.smoke()`` and the benchmark's CPU baseline leg
compare the CUDA path against.  Nothing in the product path may import it, and
it imports nothing from the product package: the two share only the seeded
input generators in ``synth``.

Modules
-------
numerics  bf16 rounding, RMSNorm, RoPE tables, SiLU (fp64 unless noted)
model     LLaMA-style decoder forward; tree-node logits defined as the causal
          forward of prompt + path (Sec. 3.3 "Tree-based Attention", App. A.3.1)
trie      valid-item prefix tree for constrained generation (Sec. 3.1)
beam      constrained log-softmax, candidate expansion, exact top-K (Sec. 2)
philox    Philox4x32-10 counter-based generator (Salmon et al., SC'11)
sd        drafting (Eq. 1), strict top-K verification (Alg. 1), relaxed
          sampling verification (Sec. 3.2, Alg. 2), the SD loop and plain
          target beam search

Parity status: every function is pinned by a ``-m "not gpu"`` test in
``tests/test_oracle_*.py`` (closed forms, brute force on tiny inputs, the
worked tree example of App. A.3.1 Table 6, statistical invariants of Eq. 4).
"""
