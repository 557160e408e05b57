// Instantiations of select_kernel (bf16 features, tensor-core update); compiled as a translation unit of
// its own so that the kernel variants build in parallel.
#include "select_impl.cuh"

namespace last {

void *select_pick_bf16_tc(int nch) {
  switch (nch) {
    case 1: return (void *)select_kernel<__nv_bfloat16, 1, 2, true>;
    case 2: return (void *)select_kernel<__nv_bfloat16, 2, 2, true>;
    case 3: return (void *)select_kernel<__nv_bfloat16, 3, 2, true>;
    case 4: return (void *)select_kernel<__nv_bfloat16, 4, 2, true>;
    case 5: return (void *)select_kernel<__nv_bfloat16, 5, 2, true>;
    case 6: return (void *)select_kernel<__nv_bfloat16, 6, 2, true>;
    case 7: return (void *)select_kernel<__nv_bfloat16, 7, 2, true>;
    case 8: return (void *)select_kernel<__nv_bfloat16, 8, 2, true>;
  }
  return nullptr;
}

}  // namespace last
