// mc_profile.h -- optional per-kernel CUDA-event timing of the library's own
// launches (enabled with mc_profile_enable; off by default, no cost when off).
#pragma once
#include <cuda_runtime.h>

namespace mc {

enum KernelId {
    kKRoute = 0,
    kKPermute,
    kKGemvW13,
    kKGemvW2,
    kKCombine,
    kKFragX,      // decode path: activations -> vector blocks
    kKGemmW13,
    kKGemmW2,
    kKRmsnorm,
    kKImportance,
    kKXImg,       // prefill path: activations -> SW128 images
    kKCount
};

bool profile_on();
// Record an event pair around one launch on `st`; call begin before and end
// after the launch.  No-ops when profiling is off.
void profile_begin(int id, cudaStream_t st);
void profile_end(int id, cudaStream_t st);

}  // namespace mc
