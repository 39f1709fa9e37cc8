"""fp64 CPU oracle for the DBLast draft+verify step.

TEST INFRASTRUCTURE ONLY.  This package checks the CUDA library; it is never
part of the product path.  Only tests/, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it.  It shares no code with the
CUDA library and imports nothing from it.

Modules: ``philox`` (Philox4x32-10 and the decision uniforms) and
``dblast_oracle`` (the step, written from the paper's definitions).
"""
