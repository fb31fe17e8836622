"""libtula_ags: the data-parallel AGS optimizer step of Tula (arXiv 2603.18112) on one GB300.

The compute path is a C-ABI CUDA library (``csrc/``, declared in
``include/tula_ags.h``); ``paper_2603_18112_gb300.tula_ags`` is its thin ctypes
binding.  ``workloads`` holds the seeded synthetic inputs.  Importing this
package loads nothing; the binding loads the library on first use and raises
if it has not been built.
"""
