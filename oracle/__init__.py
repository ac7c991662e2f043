"""CPU oracle of the ASD verifier. Test infrastructure only: the CUDA library never imports it."""
