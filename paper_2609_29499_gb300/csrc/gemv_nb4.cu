// GEMV kernels for 4 activation vectors per weight pass.
#include "gemv.cuh"

namespace tasp {
namespace gemv {

template <>
Fn pick<4>(int mode, int R, int XC) {
    return pick_nb<4>(mode, R, XC);
}

template <>
SegFn seg_pick<4>(int R) {
    return seg_pick_nb<4>(R);
}

}  // namespace gemv
}  // namespace tasp
