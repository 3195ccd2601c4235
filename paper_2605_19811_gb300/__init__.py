"""GB300 (sm_103a) LionMuon optimizer step: CUDA library + thin Python binding.

The compute path is ``liblionmuon.so`` (``csrc/``), reached through the C ABI
in ``include/lionmuon.h``; ``lionmuon`` holds the ctypes binding and ``synth``
the seeded synthetic inputs."""

from . import build, synth  # noqa: F401

__all__ = ["build", "synth"]
