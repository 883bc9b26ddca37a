// step_static.cu -- bkt_lstm_ctc_step_static: the training step for callers
// that cannot allocate device memory.  The workspace lives in one file-scope
// device array of BKT_STATIC_SCRATCH_BYTES; every GPU that loads the library
// holds that array until the process exits.
#include <mutex>

#include "bkt_internal.h"

namespace {

static __device__ __align__(256) unsigned char g_step_scratch[BKT_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
struct DeviceScratch {
  void *ptr;  // device address of g_step_scratch on this device
  int sm_count;
  bool ready;
};
DeviceScratch g_devs[kMaxDevices];
std::mutex g_devs_mu;

}  // namespace

extern "C" int bkt_lstm_ctc_step_static(const bkt_model_cfg *cfg, const bkt_batch *batch, const float *params,
                                        float *grads, float *loss, void *stream) {
  // NULL arguments are refused before any CUDA call, as by bkt_lstm_ctc_step
  if (!cfg || !batch || !params || !grads || !loss)
    return bkt::report_error(BKT_EINVAL, "bkt_lstm_ctc_step_static: NULL argument");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess)
    return bkt::report_error(BKT_ECUDA, "cudaGetDevice: %s (%s)", cudaGetErrorName(e), cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices)
    return bkt::report_error(BKT_EINVAL, "bkt_lstm_ctc_step_static: device %d out of range", dev);
  if (stream) {
    // the work goes to the stream's device: it must be the current one,
    // whose copy of the array is used (checked before anything is enqueued)
    int sdev = -1;
    e = cudaStreamGetDevice((cudaStream_t)stream, &sdev);
    if (e != cudaSuccess)
      return bkt::report_error(BKT_ECUDA, "cudaStreamGetDevice: %s (%s)", cudaGetErrorName(e), cudaGetErrorString(e));
    if (sdev != dev)
      return bkt::report_error(BKT_EINVAL,
                               "bkt_lstm_ctc_step_static: the stream belongs to device %d but device %d is current",
                               sdev, dev);
  }
  {
    // the index block goes up from one shared pageable buffer: a captured
    // copy would read whatever that buffer holds when the graph is replayed
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    e = cudaStreamIsCapturing((cudaStream_t)stream, &cs);
    if (e != cudaSuccess)
      return bkt::report_error(BKT_ECUDA, "cudaStreamIsCapturing: %s (%s)", cudaGetErrorName(e), cudaGetErrorString(e));
    if (cs != cudaStreamCaptureStatusNone)
      return bkt::report_error(BKT_EINVAL,
                               "bkt_lstm_ctc_step_static: the stream is being captured; this entry point cannot be "
                               "part of a CUDA graph");
  }
  DeviceScratch ds;
  {
    // first call on this device (with it current): look up the array's
    // device address; host code cannot use the symbol itself as a pointer
    std::lock_guard<std::mutex> lk(g_devs_mu);
    if (!g_devs[dev].ready) {
      void *p = nullptr;
      e = cudaGetSymbolAddress(&p, g_step_scratch);
      if (e != cudaSuccess)
        return bkt::report_error(BKT_ECUDA, "cudaGetSymbolAddress(step scratch): %s (%s)", cudaGetErrorName(e),
                                 cudaGetErrorString(e));
      int sms = 0;
      e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess)
        return bkt::report_error(BKT_ECUDA, "cudaDeviceGetAttribute: %s (%s)", cudaGetErrorName(e),
                                 cudaGetErrorString(e));
      g_devs[dev].ptr = p;
      g_devs[dev].sm_count = sms;
      g_devs[dev].ready = true;
    }
    ds = g_devs[dev];
  }
  return bkt::step_on_scratch(cfg, batch, params, grads, loss, (cudaStream_t)stream, ds.ptr,
                              (size_t)BKT_STATIC_SCRATCH_BYTES, ds.sm_count);
}
