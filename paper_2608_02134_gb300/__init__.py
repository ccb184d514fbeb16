"""GB300-native (sm_103a) GMC layer-boundary compression.

``paper_2608_02134_gb300.gmc`` binds the C-ABI library ``libgmc.so``;
``paper_2608_02134_gb300.workloads`` draws the seeded synthetic inputs.
Importing the package loads nothing; the library is loaded on first use and
a missing build raises instead of falling back to anything.
"""
