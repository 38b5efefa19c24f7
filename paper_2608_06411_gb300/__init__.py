"""GB300-native implementation of MAP's inference-time visual-token pruning path.

score (predictor, Eq. 3) -> select (diversity-aware greedy, Eq. 4) -> gather.
The compute runs in the CUDA library ``libmap_gb300.so`` behind a C ABI
(``include/map_gb300.h``); ``paper_2608_06411_gb300.binding`` is its thin Python
wrapper.  Importing this package does not load the library; importing ``binding``
does, and fails loudly if it has not been built.
"""
__version__ = "0.1.0"
