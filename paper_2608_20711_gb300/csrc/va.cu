// va.cu -- device memory at a chosen virtual address, for Tier 2 replay
// (AsmEvo Sec. 3.4): a captured dispatch whose kernel arguments hold
// absolute device pointers is replayed against memory restored at the
// same virtual addresses, so nested pointers stay valid.
//
// A mapping is a virtual-address reservation at the requested address,
// one physical allocation of the device, the mapping of the two and
// read/write access for the device (the CUDA virtual memory management
// calls, reached through the runtime's driver entry points, so the library
// keeps no link-time dependency on libcuda).  Host code only.
#include <mutex>
#include <new>

#include <cuda.h>
#include <cuda_runtime.h>

#include "asmv.h"
#include "nvtx_range.h"

struct asmv_va {
  int device;
  CUdeviceptr addr;
  size_t size;
  CUmemGenericAllocationHandle handle;
};

namespace {

struct VmmApi {
  decltype(&cuMemGetAllocationGranularity) granularity = nullptr;
  decltype(&cuMemAddressReserve) reserve = nullptr;
  decltype(&cuMemAddressFree) free_va = nullptr;
  decltype(&cuMemCreate) create = nullptr;
  decltype(&cuMemRelease) release = nullptr;
  decltype(&cuMemMap) map = nullptr;
  decltype(&cuMemUnmap) unmap = nullptr;
  decltype(&cuMemSetAccess) set_access = nullptr;
  bool ok = false;
};

template <class F>
bool lookup(const char *name, F *out) {
  void *fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || fn == nullptr) {
    cudaGetLastError();
    return false;
  }
  *out = reinterpret_cast<F>(fn);
  return true;
}

const VmmApi &api() {
  static VmmApi a;
  static std::once_flag once;
  std::call_once(once, [] {
    a.ok = lookup("cuMemGetAllocationGranularity", &a.granularity) &&
           lookup("cuMemAddressReserve", &a.reserve) && lookup("cuMemAddressFree", &a.free_va) &&
           lookup("cuMemCreate", &a.create) && lookup("cuMemRelease", &a.release) &&
           lookup("cuMemMap", &a.map) && lookup("cuMemUnmap", &a.unmap) &&
           lookup("cuMemSetAccess", &a.set_access);
  });
  return a;
}

CUmemAllocationProp device_prop(int device) {
  CUmemAllocationProp prop = {};
  prop.type = CU_MEM_ALLOCATION_TYPE_PINNED;
  prop.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
  prop.location.id = device;
  return prop;
}

// Make `device` current with its primary context initialised.
bool enter_device(int device, int *prev) {
  if (cudaGetDevice(prev) != cudaSuccess) *prev = -1;
  if (cudaSetDevice(device) != cudaSuccess || cudaFree(nullptr) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return true;
}

int status_of(CUresult r) {
  return r == CUDA_ERROR_OUT_OF_MEMORY ? ASMV_ENOMEM : ASMV_ECUDA;
}

}  // namespace

extern "C" {

int asmv_va_granularity(int device, size_t *out) {
  if (out == nullptr) return ASMV_EINVAL;
  int prev;
  if (!enter_device(device, &prev)) return ASMV_ECUDA;
  const VmmApi &a = api();
  int rc = ASMV_ECUDA;
  if (a.ok) {
    CUmemAllocationProp prop = device_prop(device);
    size_t g = 0;
    if (a.granularity(&g, &prop, CU_MEM_ALLOC_GRANULARITY_MINIMUM) == CUDA_SUCCESS && g > 0) {
      *out = g;
      rc = ASMV_OK;
    }
  }
  if (prev >= 0) cudaSetDevice(prev);
  return rc;
}

int asmv_va_map(int device, uint64_t addr, size_t bytes, asmv_va **out) {
  ASMV_NVTX_RANGE("asmv_va_map");
  if (out == nullptr || bytes == 0) return ASMV_EINVAL;
  int prev;
  if (!enter_device(device, &prev)) return ASMV_ECUDA;
  const VmmApi &a = api();
  int rc = ASMV_ECUDA;
  CUdeviceptr va = 0;
  size_t size = 0;
  CUmemGenericAllocationHandle h = 0;
  bool reserved = false, created = false, mapped = false;
  do {
    if (!a.ok) break;
    CUmemAllocationProp prop = device_prop(device);
    size_t g = 0;
    if (a.granularity(&g, &prop, CU_MEM_ALLOC_GRANULARITY_MINIMUM) != CUDA_SUCCESS || g == 0) break;
    if (addr % g != 0 || bytes > SIZE_MAX - g) { rc = ASMV_EINVAL; break; }
    size = (bytes + g - 1) / g * g;
    CUresult r = a.reserve(&va, size, 0, (CUdeviceptr)addr, 0);
    if (r != CUDA_SUCCESS) { rc = status_of(r); break; }
    reserved = true;
    if (addr != 0 && va != (CUdeviceptr)addr) { rc = ASMV_EINVAL; break; }   // range in use
    if ((r = a.create(&h, size, &prop, 0)) != CUDA_SUCCESS) { rc = status_of(r); break; }
    created = true;
    if ((r = a.map(va, size, 0, h, 0)) != CUDA_SUCCESS) { rc = status_of(r); break; }
    mapped = true;
    CUmemAccessDesc acc = {};
    acc.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    acc.location.id = device;
    acc.flags = CU_MEM_ACCESS_FLAGS_PROT_READWRITE;
    if ((r = a.set_access(va, size, &acc, 1)) != CUDA_SUCCESS) { rc = status_of(r); break; }
    asmv_va *m = new (std::nothrow) asmv_va;
    if (m == nullptr) { rc = ASMV_ENOMEM; break; }
    m->device = device;
    m->addr = va;
    m->size = size;
    m->handle = h;
    *out = m;
    rc = ASMV_OK;
  } while (false);
  if (rc != ASMV_OK) {
    if (mapped) a.unmap(va, size);
    if (created) a.release(h);
    if (reserved) a.free_va(va, size);
  }
  if (prev >= 0) cudaSetDevice(prev);
  return rc;
}

uint64_t asmv_va_address(const asmv_va *va) { return va ? (uint64_t)va->addr : 0; }

size_t asmv_va_size(const asmv_va *va) { return va ? va->size : 0; }

int asmv_va_unmap(asmv_va *va) {
  ASMV_NVTX_RANGE("asmv_va_unmap");
  if (va == nullptr) return ASMV_EINVAL;
  int prev;
  if (!enter_device(va->device, &prev)) return ASMV_ECUDA;
  const VmmApi &a = api();
  int rc = ASMV_ECUDA;
  if (a.ok) {
    // work still queued on this memory must finish before it disappears
    if (cudaDeviceSynchronize() == cudaSuccess && a.unmap(va->addr, va->size) == CUDA_SUCCESS &&
        a.release(va->handle) == CUDA_SUCCESS && a.free_va(va->addr, va->size) == CUDA_SUCCESS) {
      delete va;
      rc = ASMV_OK;
    }
  }
  if (prev >= 0) cudaSetDevice(prev);
  return rc;
}

}  // extern "C"
