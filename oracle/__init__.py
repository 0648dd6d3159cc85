"""CPU oracle of the MoE layer forward.

Test infrastructure only: the tests, the smoke check and the benchmark's CPU
baseline leg may import it; the product library never does.
"""
