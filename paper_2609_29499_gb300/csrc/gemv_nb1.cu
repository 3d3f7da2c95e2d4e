// GEMV kernels for 1 activation vector per weight pass.
#include "gemv.cuh"

namespace tasp {
namespace gemv {

template <>
Fn pick<1>(int mode, int R, int XC, bool gs) {
    return pick_nb<1>(mode, R, XC, gs);
}

}  // namespace gemv
}  // namespace tasp
