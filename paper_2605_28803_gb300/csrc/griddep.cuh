// Programmatic dependent launch: a kernel launched with programmatic stream serialization may
// start while the previous kernel of its stream is still running.  It must call griddep_wait()
// before any access to global memory that the previous kernel writes or reads (its inputs, and
// every output it writes); griddep_launch_dependents() lets the next kernel start early.  Both
// are no-ops for an ordinary launch.
#pragma once

namespace qvla {

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" :::); }

}  // namespace qvla
