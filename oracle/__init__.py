"""CPU oracle for the STaR-Quant SGAT W4A4 linear and TAC (test infrastructure).

This package is test infrastructure, not product code. Only the test suite,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / ``--impl reference`` legs
of ``bench.py`` may import it. The CUDA library and its Python binding never
import, link or call anything in here, and this package imports nothing from
them: the two paths share no code. Inputs reach both from the seeded
generators in ``paper_2606_04945_gb300.inputs``, which hold no arithmetic of
the method.

Every function is a plain, slow restatement of the paper:

* ``sgat``: Sec. 3.1 (Eq. 1-6) quantisers and the quantised linear, Sec. 3.2
  (Eq. 7-13) the state-guided activation transform with its literal
  split / transform / quantise / scatter, App. B weight folding.
* ``tac``: Sec. 3.3 (Eq. 17) and App. C block-wise affine compensation, and
  the App. C closed-form calibration (statistics, damping, matrix powers,
  singular-value smoothing, identity shrinkage, bias).
* ``attention``: the quantised softmax-value product of Sec. 3.3 (Z_hat,
  8-bit per-row P and 4-bit per-channel V: readings, the paper fixes
  neither) and TAC on it, one block per head; grouped-query heads.
* ``glue``: the block's glue around the quantised linears (RMSNorm, rotary
  embedding, SwiGLU), standard definitions of the model family, not the
  paper's method.

Floating point: the transform and the quantiser decision run in float32, the
precision the CUDA kernels take the integer decision in (a quantised code is
an integer decided by floating point, so both sides decide it in the same
precision). Integer GEMMs are exact. Dequantisation, TAC and calibration run
in float64.

Pins: each function is checked in ``tests/test_oracle_pins.py`` against
closed forms, brute force on tiny inputs, hand-worked fixtures in
``tests/golden/`` and the identities of App. A. No function here is
"parity unpinned".
"""

from . import attention, glue, sgat, tac  # noqa: F401
