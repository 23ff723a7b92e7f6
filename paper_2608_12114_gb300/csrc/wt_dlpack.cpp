// The file-backed tensor producer (Algorithm 1, Sec. 7.1) for CUDA: a read-only shared
// mapping of a file range, exposed to the device and wrapped in a versioned DLPack capsule
// whose deleter owns the mapping.  See include/wt_dlpack.h for the contract.
//
// Device exposure on this platform (Sec. 7.3, the route probe of wt_open): where the GPU
// reads pageable memory through the host page tables, the capsule's data pointer is the
// mapping itself; otherwise the range is host-registered (mapped; read-only where the
// driver accepts it) and the capsule carries the registration's device pointer.
#include <fcntl.h>
#include <sys/mman.h>
#include <sys/stat.h>
#include <unistd.h>

#include <atomic>
#include <cerrno>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>

#include <cuda_runtime.h>

#include "../../include/wt_dlpack.h"
#include "wt_kernels.h"

namespace {

std::atomic<int64_t> g_live{0};

struct Ctx {
  void *map = nullptr;
  size_t map_len = 0;
  bool registered = false;
  int64_t shape[4] = {0, 0, 0, 0};
  int64_t strides[4] = {0, 0, 0, 0};
  DLManagedTensorVersioned mt;
};

// The capsule's deleter: Release (unregister) then munmap, as in Algorithm 1's last step.
void ctx_deleter(DLManagedTensorVersioned *self) {
  if (!self) return;
  Ctx *c = static_cast<Ctx *>(self->manager_ctx);
  if (c->registered) {
    cudaHostUnregister(c->map);
    cudaGetLastError();
  }
  munmap(c->map, c->map_len);
  delete c;
  g_live.fetch_sub(1, std::memory_order_relaxed);
}

int err(int code, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
int err(int code, const char *fmt, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  return wt::set_error(code, buf);
}

bool dl_dtype(int32_t dtype, DLDataType *t, uint32_t *esz) {
  switch (dtype) {
    case WT_F32: *t = {kDLFloat, 32, 1}; *esz = 4; return true;
    case WT_BF16: *t = {kDLBfloat, 16, 1}; *esz = 2; return true;
    case WT_F16: *t = {kDLFloat, 16, 1}; *esz = 2; return true;
    case WT_I8: *t = {kDLInt, 8, 1}; *esz = 1; return true;
    case WT_U8: *t = {kDLUInt, 8, 1}; *esz = 1; return true;
    default: return false;
  }
}

}  // namespace

namespace wt {

int dlpack_map(const char *path, uint64_t off, uint64_t nbytes, int32_t dtype, int ndim, const uint64_t *shape,
               unsigned flags, DLManagedTensorVersioned **out) {
  DLDataType dt;
  uint32_t esz;
  if (!dl_dtype(dtype, &dt, &esz)) return err(WT_EINVAL, "dlpack: dtype %d", (int)dtype);
  if (ndim < 1 || ndim > 4) return err(WT_EINVAL, "dlpack: ndim %d", ndim);
  if (nbytes == 0) return err(WT_EINVAL, "dlpack: %s: zero-byte tensor", path);
  if (flags & ~WT_DLPACK_HOST) return err(WT_EINVAL, "dlpack: unknown flag bits 0x%x", flags);
  const uint64_t page = (uint64_t)sysconf(_SC_PAGESIZE);
  const uint64_t a0 = off / page * page;
  const uint64_t len = (off + nbytes + page - 1) / page * page - a0;
  const int fd = open(path, O_RDONLY | O_CLOEXEC);
  if (fd < 0) return err(WT_EIO, "dlpack: open %s: %s", path, strerror(errno));
  const bool injected = wt::fault_injected("mmap");
  void *p = injected ? MAP_FAILED : mmap(nullptr, len, PROT_READ, MAP_SHARED, fd, (off_t)a0);
  const int e = errno;
  close(fd);  // the mapping keeps the file referenced
  if (p == MAP_FAILED) return err(WT_EIO, "dlpack: mmap %s: %s", path, injected ? "injected fault" : strerror(e));
  Ctx *c = new (std::nothrow) Ctx();
  if (!c) {
    munmap(p, len);
    return err(WT_ENOMEM, "dlpack: out of host memory");
  }
  c->map = p;
  c->map_len = len;
  uint8_t *data = static_cast<uint8_t *>(p) + (off - a0);
  DLDevice dev = {kDLCPU, 0};
  if (!(flags & WT_DLPACK_HOST)) {
    int d = 0;
    cudaError_t ce = cudaGetDevice(&d);
    int ats = 0;
    if (ce == cudaSuccess) ce = cudaDeviceGetAttribute(&ats, cudaDevAttrPageableMemoryAccessUsesHostPageTables, d);
    if (ce != cudaSuccess) {
      munmap(p, len);
      delete c;
      cudaGetLastError();
      return err(WT_ECUDA, "dlpack: %s", cudaGetErrorString(ce));
    }
    if (!ats) {
      ce = cudaHostRegister(p, len, cudaHostRegisterMapped | cudaHostRegisterReadOnly);
      if (ce != cudaSuccess) {
        cudaGetLastError();
        ce = cudaHostRegister(p, len, cudaHostRegisterMapped);
      }
      void *dp = nullptr;
      if (ce == cudaSuccess) {
        c->registered = true;
        ce = cudaHostGetDevicePointer(&dp, p, 0);
      }
      if (ce != cudaSuccess) {
        cudaGetLastError();
        if (c->registered) cudaHostUnregister(p);
        munmap(p, len);
        delete c;
        return err(WT_ENOTSUP, "dlpack: %s: the device cannot read these host pages (%s)", path,
                   cudaGetErrorString(ce));
      }
      data = static_cast<uint8_t *>(dp) + (off - a0);
    }
    dev = {kDLCUDA, d};
  }
  int64_t stride = 1;
  for (int k = ndim - 1; k >= 0; --k) {
    c->shape[k] = (int64_t)shape[k];
    c->strides[k] = stride;
    stride *= (int64_t)shape[k];
  }
  DLManagedTensorVersioned &mt = c->mt;
  mt.version = {1, 0};
  mt.manager_ctx = c;
  mt.deleter = ctx_deleter;
  mt.flags = DLPACK_FLAG_BITMASK_READ_ONLY;
  mt.dl_tensor.data = data;
  mt.dl_tensor.device = dev;
  mt.dl_tensor.ndim = ndim;
  mt.dl_tensor.dtype = dt;
  mt.dl_tensor.shape = c->shape;
  mt.dl_tensor.strides = c->strides;
  mt.dl_tensor.byte_offset = 0;
  g_live.fetch_add(1, std::memory_order_relaxed);
  *out = &mt;
  return WT_OK;
}

}  // namespace wt

#pragma GCC visibility push(default)
extern "C" {

int wt_dlpack_file(const char *path, int32_t dtype, uint64_t M, uint64_t K, unsigned flags,
                   DLManagedTensorVersioned **out) {
  if (!out) return err(WT_EINVAL, "wt_dlpack_file: out is NULL");
  *out = nullptr;
  if (!path) return err(WT_EINVAL, "wt_dlpack_file: path is NULL");
  DLDataType dt;
  uint32_t esz;
  if (!dl_dtype(dtype, &dt, &esz)) return err(WT_EINVAL, "wt_dlpack_file: dtype %d", (int)dtype);
  struct stat st;
  if (stat(path, &st) != 0) return err(WT_EIO, "wt_dlpack_file: stat %s: %s", path, strerror(errno));
  const uint64_t n = (uint64_t)st.st_size;
  const uint64_t page = (uint64_t)sysconf(_SC_PAGESIZE);
  unsigned __int128 want = (unsigned __int128)M * K * esz;
  if (want != n) return err(WT_EINVAL, "wt_dlpack_file: %s: rejected, %llu bytes but M*K*sizeof = %llu", path,
                            (unsigned long long)n, (unsigned long long)(uint64_t)want);
  if (n == 0 || n % page != 0)
    return err(WT_EINVAL, "wt_dlpack_file: %s: rejected, size %llu is not a non-zero multiple of the page size %llu",
               path, (unsigned long long)n, (unsigned long long)page);
  const uint64_t shape[2] = {M, K};
  return wt::dlpack_map(path, 0, n, dtype, 2, shape, flags, out);
}

void wt_dlpack_release(DLManagedTensorVersioned *t) {
  if (t && t->deleter) t->deleter(t);
}

int wt_dlpack_live(int64_t *n) {
  if (!n) return err(WT_EINVAL, "wt_dlpack_live: NULL argument");
  *n = g_live.load(std::memory_order_relaxed);
  return WT_OK;
}

}  // extern "C"
#pragma GCC visibility pop
