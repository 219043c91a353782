"""Trident SCM on GB300: a guarded-dispatch C-ABI library (sm_103a kernels) and its
thin Python binding. `scm` is the binding; `synth` draws seeded synthetic inputs."""
