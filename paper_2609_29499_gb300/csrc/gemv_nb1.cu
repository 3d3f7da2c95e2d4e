// GEMV kernels for 1 activation vector per weight pass.
#include "gemv.cuh"

namespace tasp {
namespace gemv {

template <>
Fn pick<1>(int mode, int R, int XC) {
    return pick_nb<1>(mode, R, XC);
}

template <>
SegFn seg_pick<1>(int R) {
    return seg_pick_nb<1>(R);
}

}  // namespace gemv
}  // namespace tasp
