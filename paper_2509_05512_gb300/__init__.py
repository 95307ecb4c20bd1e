"""GB300-native quaternion convolution forward (QUAN, arXiv 2509.05512).

The compute path is the CUDA library ``libquan`` (sm_103a); ``quan`` holds the
thin ctypes binding and ``inputs`` the seeded synthetic input generators.
"""
