"""GB300-native SMoES router hot path (modality-guided MoE routing with inter-bin MI).

The compute path is the CUDA library ``lib/libsmoes.so`` (built by ``build.build_library``)
behind the C ABI declared in ``include/smoes.h``; ``binding`` marshals arguments to it.
"""
