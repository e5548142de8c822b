"""WISE attention hot path on GB300 (sm_103a).

The compute path is the C-ABI library libwise.so built from csrc/ (three
hand-written CUDA kernels: dense causal attention with a fused block-mass
epilogue, support selection, support-restricted sparse attention).
`paper_2609_27373_gb300.wise` is the thin ctypes binding with the same names
as the C entry points; `synth` draws seeded synthetic inputs.
"""
