"""GB300-native trie-automaton token masks for constrained decoding.

The compute path lives in the CUDA library ``libtriemask.so`` (C ABI declared
in ``include/triemask.h``); ``triemask`` is its thin ctypes binding. Importing
this package loads nothing; the binding loads the library on first use and
raises if it has not been built.
"""
