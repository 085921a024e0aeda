// nvtx_range.h -- one NVTX range per C ABI call, in the "asmv" domain, so that
// a profiler's timeline shows each call (its host-side validation and packing,
// its launches and its readback) under the call's name.  NVTX3 is header-only:
// without a profiler attached, a range costs a branch on a null callback.
#pragma once
#include <cstring>

#include <nvtx3/nvToolsExt.h>

namespace asmv {

inline nvtxDomainHandle_t nvtx_domain() {
  static const nvtxDomainHandle_t d = nvtxDomainCreateA("asmv");
  return d;
}

class NvtxRange {
 public:
  explicit NvtxRange(const char *name) {
    nvtxEventAttributes_t a;
    std::memset(&a, 0, sizeof a);
    a.version = NVTX_VERSION;
    a.size = NVTX_EVENT_ATTRIB_STRUCT_SIZE;
    a.messageType = NVTX_MESSAGE_TYPE_ASCII;
    a.message.ascii = name;
    nvtxDomainRangePushEx(nvtx_domain(), &a);
  }
  ~NvtxRange() { nvtxDomainRangePop(nvtx_domain()); }
  NvtxRange(const NvtxRange &) = delete;
  NvtxRange &operator=(const NvtxRange &) = delete;
};

}  // namespace asmv

#define ASMV_NVTX_RANGE(name) ::asmv::NvtxRange asmv_nvtx_range_(name)
