"""CPU oracle for the low-bit recurrent-state method (test infrastructure only).

Only the test-suite, ``__graft_entry__.smoke()`` and the benchmark's ``cpu_baseline`` /
``--impl reference`` legs may import this package.  The product library never does.
"""
