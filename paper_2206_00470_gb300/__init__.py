"""GB300 parameter manager driven by intent signals (AdaPM, arXiv 2206.00470).

The compute path is libadapm.so (CUDA kernels for sm_103a behind the C ABI in
include/adapm.h); ``adapm`` is its thin Python binding and ``build`` compiles
it.  Importing the package loads nothing: ``adapm.load()`` (or creating a
``ParameterManager``) loads the library and fails loudly if it is missing.
"""
