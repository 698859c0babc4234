"""CPU oracle for the low-bit KV decode step and the DGAP epilogue.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call or
execute this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.

It is a plain, slow, obviously correct restatement of the method in numpy
(float64 wherever the method is floating point, IEEE float32 single
operations where the stored format fixes float32 rounding).  It shares no
code with the CUDA path.  Every function cites the section / equation of the
paper (arXiv 2607.16248, "High-accuracy Low-Bit KV-Cache Quantization via
Local Distribution Restoration") that it follows, or names the reading taken
where the paper is silent.

Modules
-------
quant      asymmetric b-bit group quantizer, bit packing, residual window
attention  GQA decode attention softmax(q K^T / sqrt(d)) V over the cache
dgap       top-K window, risk features, detector, gate, corrector, merge
drift      offline drift metrics (C(alpha), c_t, d_loc, y_t) and the K_b rule
"""

from . import quant, attention, dgap, drift  # noqa: F401
