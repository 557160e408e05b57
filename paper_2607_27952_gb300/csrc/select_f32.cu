// Instantiations of select_kernel (fp32 features, CUDA-core update); compiled as a translation unit of
// its own so that the kernel variants build in parallel.
#include "select_impl.cuh"

namespace last {

void *select_pick_f32(int nch) {
  switch (nch) {
    case 1: return (void *)select_kernel<float, 1, 2, false>;
    case 2: return (void *)select_kernel<float, 2, 2, false>;
    case 3: return (void *)select_kernel<float, 3, 2, false>;
    case 4: return (void *)select_kernel<float, 4, 2, false>;
    case 5: return (void *)select_kernel<float, 5, 2, false>;
    case 6: return (void *)select_kernel<float, 6, 2, false>;
    case 7: return (void *)select_kernel<float, 7, 2, false>;
    case 8: return (void *)select_kernel<float, 8, 2, false>;
  }
  return nullptr;
}

}  // namespace last
