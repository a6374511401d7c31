"""fp64 CPU oracle for the KV-COBRA hot path (arXiv 2609.24298).

TEST INFRASTRUCTURE ONLY.  Only `tests/`, `__graft_entry__.smoke()` and the
`cpu_baseline` / `--impl reference` legs of `bench.py` may import this package.  The
product (the C-ABI library and its Python binding) never calls it and shares no code
with it.

Every function restates, in plain slow numpy, a step the paper defines; each cites the
section / equation / table it follows.  Where the paper is silent or ambiguous the
reading taken is stated in the docstring.

Modules
  hadamard   fused Walsh-Hadamard rotation with the random sign flip (Sec. 3.4)
  quantizer  Bennett distortion q(b), the static uniform scalar quantizer, loading factor
  allocator  head distortion D(r,b), C1, C2 damped update, exact DP, brute force
  calibrate  centred covariance, eigenbasis, attention-KL weights and reordering, basis fusion
  layout     the packed code-row layout (bit position of every code)
  attention  dequantise-on-read decode attention, plain definition and rank-space algebra
  rope       decode with the rotary embedding applied to the reconstructed keys and the query
  compress   per-token projection + quantisation (Table alg:kvrobin step 7)
  measured   App. E's measured per-head distortion tables and the exact DP over them

Parity status: the damped C2 update is a heuristic with no optimality guarantee
(App. D says so itself); its output is pinned only through invariants - "parity unpinned"
for optimality.  Everything else is pinned by tests/test_oracle_*.py.
"""
