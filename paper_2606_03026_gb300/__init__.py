"""GB300-native spike-gated INT8 projection (sm_103a CUDA behind a C ABI).

``y = s * (Q x)`` for binary spikes ``x``, column-major INT8 ``Q`` and FP32
per-output-channel scales ``s`` (Section 2.3, Eq. sparse).  The compute runs in
``libspikeproj.so``; :mod:`.spikeproj` is its ctypes binding and
:mod:`.synth` makes seeded synthetic inputs.  Importing the package loads
nothing: the library is opened on first use and a missing build is an error.
"""
__all__ = ["spikeproj", "synth"]
