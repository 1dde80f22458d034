"""CPU oracle for the MINW-Net inference path and the AQE quantizer.

TEST INFRASTRUCTURE ONLY: a plain, slow, deterministic restatement of the
paper's definitions that the CUDA path is checked against.  Only tests/,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` leg of ``bench.py`` may
import it.  It shares no code with the CUDA library and never loads it.
"""
