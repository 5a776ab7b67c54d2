"""TRACK oracle: a plain, slow, fp64 CPU restatement of the routed-denoising hot path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, links or runs
this package.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline and reference legs may use it.  It shares no code with the CUDA
library (``paper_2609_30096_gb300``); the one module both sides use is the
seeded input generator ``synth``, which holds no arithmetic of the method.

Contents (each function cites the passage of the paper it restates):

* ``oracle.track`` - the method proper: guidance (Eq. 1), the scheduler update
  (Eq. 2: the flow-matching Euler instance, and a second-order multistep
  instance whose history h_i carries across model switches), routed sampling
  (Eq. 3), the relative disagreement (Eq. 4) and its frequency-band split
  (Sec. 4.4), the mean score (Eq. 5), the box-constrained relaxation and its
  threshold solution (Eq. 6-7), top-K switching (Sec. 3.2.3), the equal-budget
  First-K / Last-K / Random-K policies (Sec. 4.5) and reference-trajectory
  calibration (Sec. 3.2.1).
* ``oracle.dit`` - the denoiser f_m that Eq. 1 treats as a black box: the
  Wan-style video DiT (patchify, adaLN-modulated self-attention with 3D RoPE,
  cross-attention, GELU MLP, unpatchify).  The paper does not define these
  internals (Sec. 3.1 says only that the pair shares latent, output shape,
  conditioning interface and prediction target); the definitions written here
  are this library's reading, pinned by component tests (closed forms,
  invariants, brute force) and by structural tests of the composed block.
  ``DiT.forward_at_tokens`` evaluates the last block and the head at chosen
  tokens only, for checks at sizes where the whole forward is too slow.

Precision: everything is computed in fp64 from fp32 inputs.  ``precision="bf16"``
rounds the weight matrices and the text conditioning to bf16 (round to nearest
even) before the same fp64 arithmetic, which is what the GPU's bf16 mode feeds
its tensor cores; the GPU additionally rounds activations, which the parity
tolerance covers.

Parity status: every function of ``oracle.track`` is pinned by closed forms,
invariants and brute force.  The DiT as a whole has no worked example in the
paper ("parity unpinned" by the paper); it is pinned by its components and by
the structural block tests in ``tests/test_oracle_dit.py``.
"""

from . import dit, track  # noqa: F401
