"""VaSE eviction step on GB300 (sm_103a): C-ABI library + thin Python binding.

The CUDA library is ``_lib/libvase.so`` (built by ``paper_2606_03928_gb300.build``);
``paper_2606_03928_gb300.vase`` mirrors its entry points with the same names, and
``paper_2606_03928_gb300.workloads`` draws the seeded synthetic inputs.
"""
