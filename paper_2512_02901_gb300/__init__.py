"""GB300-native Fairy2i widely-linear {+-1, +-i} layer: a C-ABI CUDA library (sm_103a) and a
thin ctypes binding. Importing the package loads nothing; the library is opened on first use
and a missing library raises (there is no CPU fallback)."""
