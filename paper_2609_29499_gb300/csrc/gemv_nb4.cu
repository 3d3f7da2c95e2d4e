// GEMV kernels for 4 activation vectors per weight pass.
#include "gemv.cuh"

namespace tasp {
namespace gemv {

template <>
Fn pick<4>(int mode, int R, int XC, bool gs) {
    return pick_nb<4>(mode, R, XC, gs);
}

}  // namespace gemv
}  // namespace tasp
