"""Bit-precise SAMD arithmetic on GB300 (sm_103a).

The compute path is the C-ABI library ``libsamd.so`` (hand-written CUDA);
``paper_1809_10572_gb300.samd`` is its thin Python binding. Importing the
package itself loads nothing, so the CPU-only tests can use ``synth``.
"""
__all__ = ["samd", "synth"]
