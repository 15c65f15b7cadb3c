"""Seeded synthetic inputs shared by the tests, the bench and the oracle
harness: value generators, layout descriptions and buffer materialisation.
Nothing here computes the reshuffle, its volumes or its relabeling."""
