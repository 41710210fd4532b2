"""GB300-native (sm_103a) Flash-BoN draft-generation path.

`flashbon` is the ctypes binding of the C-ABI library libflashbon.so (built by
`paper_2607_04461_gb300.build`); `synth` generates seeded synthetic inputs.
The binding is imported lazily so that `synth` works without the library.
"""
__all__ = ["flashbon", "synth", "build"]
