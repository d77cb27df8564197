"""AsymSpec per-step fuse-and-verify on GB300 (sm_103a)."""
