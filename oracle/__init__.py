"""fp64 CPU oracle for causal / document-masked attention (test infrastructure only)."""
