"""fp64 CPU oracle for Curvature-Conditioned Query (arxiv 2606.01294).

TEST INFRASTRUCTURE ONLY: the test-suite, the smoke check and the CPU-baseline
leg of the benchmark are the only callers.  The GPU library never imports,
links or executes anything here, and nothing here imports the GPU library.

The arithmetic lives in ``ccq_oracle.c`` (plain C, fp64, token by token);
this module compiles it with gcc on first use and marshals numpy arrays.

Parity status of each routine (what pins it is in ``tests/test_oracle_pins.py``):
  forward(chunk=0)   recurrent CCQ-GLA / CCQ-GDN (Algorithm 2, Eq. clean/read)
                     -- pinned by brute force, closed forms, invariants and the
                     finite-difference Hessian identity.
  forward(chunk>0)   chunkwise form (Algorithm 1, App. B) -- pinned by equality
                     with the recurrent form.
  gla_backward       reverse mode of the CCQ-GLA forward -- pinned by central
                     finite differences of the forward (fp64).
  gdn_backward       reverse mode of the CCQ-Gated-DeltaNet forward -- pinned the
                     same way (tests/test_oracle_backward_gdn.py) and by a chunkwise
                     adjoint; the reference of the ccq_gdn_bwd parity tests.
  gdn_forward_decayed  CCQ-Gated-DeltaNet with the decay-aligned covariance (a reading of
                     the paper's future-work variant, stated in ccq_oracle.c) -- pinned
                     by brute-force weighted covariances, the undecayed special case,
                     the spectrum bound and resumption (tests/test_oracle_decayed.py);
                     the reference of the ccq_gdn_fwd_decayed parity tests.
  gdn_forward_spectral  CCQ-Gated-DeltaNet with the read contracted by I - x, (I + x)^{-1}
                     or exp(-x), x = lambda Sigma (the paper's operator and the two
                     alternatives it names), undecayed or decay-aligned statistics; numpy,
                     token by token -- pinned against the C oracle (linear case), explicit
                     eigendecompositions, the first-order agreement in lambda and the
                     spectrum bounds (tests/test_oracle_spectral.py).
  Absolute outputs on the benchmark-shaped random inputs are pinned only
  through the above: the paper prints no worked numerical example.
"""
from .ccq_oracle import (  # noqa: F401
    build_oracle,
    forward,
    decode_step,
    gla_backward,
    gdn_backward,
    gdn_forward_decayed,
    gdn_forward_spectral,
    GLA,
    GDN,
    LINEAR,
    RESOLVENT,
    EXPONENTIAL,
)
