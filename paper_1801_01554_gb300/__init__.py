"""Back-propagation training step for sigmoid MLPs on GB300 (sm_103a).

The compute path is the CUDA library ``libbp.so`` behind a C ABI; ``bp`` is its
ctypes binding.  Importing this package does not load the library: the binding
loads it on first use and raises if it has not been built.
"""
