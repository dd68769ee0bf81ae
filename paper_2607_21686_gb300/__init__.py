"""GB300-native data-parallel hot path of Persistent Computational State.

``paper_2607_21686_gb300.pcs`` is the binding of the C-ABI library
``libpcs.so`` (hand-written sm_103a kernels); ``paper_2607_21686_gb300.synth``
draws the seeded synthetic session populations.  Importing the package
itself loads nothing.
"""
__all__ = ["pcs", "synth"]
