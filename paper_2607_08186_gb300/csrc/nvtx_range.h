// NVTX ranges around the C ABI entry points (host code): each call that enqueues
// device work shows up as a named range of the "hdsfa" domain in a profiler's
// timeline (ncu --nvtx, nsys).  NVTX v3 is header-only; with no tool attached a range
// costs one check of an unset function pointer.
#pragma once
#include <nvtx3/nvToolsExt.h>

namespace hdsfa {

inline nvtxDomainHandle_t nvtx_domain() {
  static nvtxDomainHandle_t d = nvtxDomainCreateA("hdsfa");
  return d;
}

class NvtxRange {
 public:
  explicit NvtxRange(const char* name) {
    nvtxEventAttributes_t a = {};
    a.version = NVTX_VERSION;
    a.size = NVTX_EVENT_ATTRIB_STRUCT_SIZE;
    a.messageType = NVTX_MESSAGE_TYPE_ASCII;
    a.message.ascii = name;
    nvtxDomainRangePushEx(nvtx_domain(), &a);
  }
  ~NvtxRange() { nvtxDomainRangePop(nvtx_domain()); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

}  // namespace hdsfa

#define HD_NVTX_RANGE(name) ::hdsfa::NvtxRange hd_nvtx_range_(name)
