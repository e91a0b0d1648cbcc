"""Seeded synthetic inputs (shapes, drift recipes, generators) shared by the
tests, the smoke check and the benchmark.  Holds none of the method's
arithmetic: it only produces weights, snapshots and Adam moments."""
