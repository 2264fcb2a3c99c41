"""GB300 (sm_103a) resettable memoroid scans over tapes of concatenated episodes.

The compute lives in the C-ABI library libmemoroid.so (include/memoroid.h);
`paper_2402_09900_gb300.memoroid` is its ctypes binding (import it directly).
"""
