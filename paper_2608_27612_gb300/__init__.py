"""GB300-native eager multi-resolution substrate discovery (EMR-HyperNEAT hot path).

The compute path lives in the C-ABI library ``libemr`` (hand-written CUDA for
sm_103a); ``paper_2608_27612_gb300.emr`` is its thin ctypes binding. Importing the
package does not load the library; the binding loads it on first use and raises
if it has not been built.
"""
