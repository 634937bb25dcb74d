"""CPU oracle of the LAEP MoE expert-layer hot path (test infrastructure only).

Only the tests, the smoke check and the benchmark's CPU-baseline leg use this
package; the CUDA library never imports it.
"""
