"""CPU oracle for the energy-guided cached DiT step (EchoCache, Sec. 3.3 and 3.4).

TEST INFRASTRUCTURE ONLY.  Plain, slow, obviously-correct numpy restatements
of what the paper defines, used to check the CUDA path.  Only `tests/`,
`__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py` may import
this package; the product package never does, and this package imports
nothing from it.  Floating point is fp64 except where a rule fixes fp32 so that
the CUDA path can be compared bit for bit (drift score, selection keys,
int8 quantisation, dequantisation): there the fp32 operations are written out
one by one in the stated order.

Modules:
  energy  - Cross-modal saliency anchors: segment STFT energy, per-segment weight.
  select  - per-token Eq. 1 drift against the cache, energy-weighted top-K.
  cache   - int8 per-token quantisation and reconstruction (Sec. 3.4).
  block   - the DiT block on active latents (Q' on active, K/V on all, FFN on
            active) and the mask fusion.
  step    - one cached layer step, the step loop, the uncached block.
  schedule - step-level Eq. 1 change and the adaptive update rate r_t.
  refcache - cache forms: plain int8, full precision (ablation), and the
            reference-plus-int8-residual manager of Sec. 3.4.

Parity status per function is stated in each module header.
"""
from . import block, cache, energy, refcache, schedule, select, step  # noqa: F401
