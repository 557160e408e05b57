// Instantiations of select_kernel (bf16 features, CUDA-core update); compiled as a translation unit of
// its own so that the kernel variants build in parallel.
#include "select_impl.cuh"

namespace last {

void *select_pick_bf16(int nch, int tb) {
  if (tb == 4) {
    switch (nch) {
      case 1: return (void *)select_kernel<__nv_bfloat16, 1, 4, false>;
      case 2: return (void *)select_kernel<__nv_bfloat16, 2, 4, false>;
      case 3: return (void *)select_kernel<__nv_bfloat16, 3, 4, false>;
      case 4: return (void *)select_kernel<__nv_bfloat16, 4, 4, false>;
      case 5: return (void *)select_kernel<__nv_bfloat16, 5, 4, false>;
      case 6: return (void *)select_kernel<__nv_bfloat16, 6, 4, false>;
      case 7: return (void *)select_kernel<__nv_bfloat16, 7, 4, false>;
      case 8: return (void *)select_kernel<__nv_bfloat16, 8, 4, false>;
    }
    return nullptr;
  }
  switch (nch) {
    case 1: return (void *)select_kernel<__nv_bfloat16, 1, 2, false>;
    case 2: return (void *)select_kernel<__nv_bfloat16, 2, 2, false>;
    case 3: return (void *)select_kernel<__nv_bfloat16, 3, 2, false>;
    case 4: return (void *)select_kernel<__nv_bfloat16, 4, 2, false>;
    case 5: return (void *)select_kernel<__nv_bfloat16, 5, 2, false>;
    case 6: return (void *)select_kernel<__nv_bfloat16, 6, 2, false>;
    case 7: return (void *)select_kernel<__nv_bfloat16, 7, 2, false>;
    case 8: return (void *)select_kernel<__nv_bfloat16, 8, 2, false>;
  }
  return nullptr;
}

}  // namespace last
