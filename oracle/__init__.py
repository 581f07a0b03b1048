"""Plain fp64 CPU oracle of the AdaDSF depth-sparse forward (test infrastructure only)."""
