"""CPU oracle for the DAMP decode-step state update (arxiv 2608.27513).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` import this package.  The product path (the
CUDA library and its binding) never imports, links or runs anything here, and
this package never imports the product path.  The two share only the seeded
input generators in ``workloads.py``.

* ``oracle.core``      -- ctypes wrapper over the plain-C oracle (damp_oracle.c):
                          FP16 conversion, H_32, the UINT8 affine quantizer, the
                          packed tiers, the FP32 delta step, the quantized step.
* ``oracle.calibrate`` -- the offline channel-selection score (error energy x
                          persistence), TopK and the stable partition (Algorithm 1),
                          in float64 numpy.
* ``oracle.runs``      -- plain drivers: FP32 prefix trajectories, calibration
                          trajectories, free-running mixed-precision trajectories.

Parity unpinned: agreement with the paper's own kernel (its min/max order,
metadata rounding and FMA use) and with its accuracy numbers; the paper prints
no worked state or output values.
"""
