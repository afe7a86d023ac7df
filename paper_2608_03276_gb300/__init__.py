"""TaskPress prefill-time KV compression on GB300 (sm_103a).

The compute path lives in the C-ABI library ``libtaskpress.so`` (CUDA kernels
under ``csrc/``); ``binding`` marshals torch tensors into it.  Importing the
package loads nothing: ``binding.load()`` does, and raises when the library
is missing.
"""
