"""LaCache's two-stage lookahead semantic-cache lookup on GB300 (sm_103a).

The product is the C-ABI library ``liblacache.so`` (CUDA kernels, declared in ``include/lacache.h``). The
``lacache`` module binds it with the same function names. ``workloads`` draws seeded synthetic inputs. Importing
the package loads nothing: the library is opened on first use of the binding, and the binding fails loudly if it
has not been built.
"""
