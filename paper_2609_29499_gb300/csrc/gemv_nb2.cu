// GEMV kernels for 2 activation vectors per weight pass.
#include "gemv.cuh"

namespace tasp {
namespace gemv {

template <>
Fn pick<2>(int mode, int R, int XC, bool gs) {
    return pick_nb<2>(mode, R, XC, gs);
}

}  // namespace gemv
}  // namespace tasp
