"""CPU oracle for StepKV's compression pass -- test infrastructure only (see stepkv_oracle)."""
