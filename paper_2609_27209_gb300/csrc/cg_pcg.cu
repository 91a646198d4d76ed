// cg_pcg.cu -- the Jacobi-preconditioned instantiations of the resident CG kernel (an optional
// solver variant, not the paper's method: M = diag(L_eps) = deg + eps, preconditioned CG as in
// Y. Saad, "Iterative Methods for Sparse Linear Systems", Algorithm 9.1).  A translation unit of
// their own, so that they compile in parallel with the plain solver.
#include "cg_device.cuh"

namespace erc {

const void* resident_kernel_pc(int nvec, bool weighted, bool ps) {
  return resident_kernel_for<true>(nvec, weighted, ps);
}

}  // namespace erc
