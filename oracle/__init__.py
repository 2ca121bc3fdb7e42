"""CPU fp64 oracle for the structured-suffix denoising step (test infrastructure only)."""
