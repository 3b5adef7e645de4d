// Programmatic dependent launch for the per-layer kernels.
//
// Every per-step kernel of the per-layer (generic) path starts with pdl_entry(): it first lets its own
// dependents launch (griddepcontrol.launch_dependents: once every CTA of this grid has issued it, the
// next kernel's CTAs may be scheduled as SMs free up), then waits (griddepcontrol.wait) until the grid
// it depends on has completed and its writes are visible.  Nothing before the wait touches memory, so a
// captured graph may turn any kernel-to-kernel edge into such a kernel into a programmatic one (every
// kernel of the library but the fused row and update kernels, which place their waits themselves): the
// dependent's launch and CTA scheduling overlap the producer's tail instead of following it.  Launched
// without a programmatic dependency, both instructions return at once.
#pragma once

namespace vfl {

__device__ __forceinline__ void pdl_entry() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

}  // namespace vfl
