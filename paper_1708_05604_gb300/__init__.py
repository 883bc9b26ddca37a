"""GB300-native bucketed LSTM-CTC training step (arXiv 1708.05604).

The compute path is the C-ABI library ``libbkt.so`` (hand-written CUDA for
sm_103a plus a host C++ planner and step engine), reached through the thin
ctypes binding in ``binding``.  Importing this package loads nothing; the
binding loads the library on first use and raises if it is missing.
"""
__all__ = ["binding", "synth"]
