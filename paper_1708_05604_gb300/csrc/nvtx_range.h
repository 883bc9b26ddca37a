// nvtx_range.h -- host-side NVTX ranges naming the step's phases and
// kernels, so that a profiler can group or filter the launches by them (for
// instance `ncu --nvtx --nvtx-include "bkt_lstm_ctc_step/lstm_bwd/"`).
// Without a profiler attached, NVTX's first call finds no tool and every
// later call returns at once.  Where the toolkit has no NVTX v3 headers the
// ranges compile to nothing.
#pragma once

#if defined(__has_include)
#if __has_include(<nvtx3/nvToolsExt.h>)
#include <nvtx3/nvToolsExt.h>
#define BKT_HAVE_NVTX 1
#endif
#endif

namespace bkt {

// A range open from construction to end() or destruction, whichever is
// first, on the calling thread.
class NvtxRange {
 public:
  explicit NvtxRange(const char *name) {
#ifdef BKT_HAVE_NVTX
    nvtxRangePushA(name);
#else
    (void)name;
#endif
  }
  void end() {
    if (open_) {
#ifdef BKT_HAVE_NVTX
      nvtxRangePop();
#endif
      open_ = false;
    }
  }
  ~NvtxRange() { end(); }
  NvtxRange(const NvtxRange &) = delete;
  NvtxRange &operator=(const NvtxRange &) = delete;

 private:
  bool open_ = true;
};

}  // namespace bkt
