/* wt_dlpack.h - the file-backed tensor producer (Algorithm 1, Sec. 7.1): a file's pages,
 * mapped read-only and shared, handed to a tensor framework as a versioned DLPack capsule
 * with no copy.  C ABI; part of libwt.so (see wt.h for the status codes and dtypes).
 *
 * The DLPack declarations below follow the published DLPack ABI (version 1.x:
 * DLManagedTensorVersioned); a consumer built against dlpack.h reads them unchanged.
 *
 * Ownership: every successful producer call returns one DLManagedTensorVersioned that owns
 * exactly one mapping (and, where the device needed one, one host registration); nothing is
 * cached across calls.  Calling its deleter (directly, through wt_dlpack_release, or by the
 * consumer that adopted it) unregisters and unmaps the range and frees the struct.  The
 * deleter touches no Python or framework state and may run on any thread.
 *
 * Read-only: the capsule carries DLPACK_FLAG_BITMASK_READ_ONLY.  DLPack leaves enforcement
 * to the consumer; the pages are mapped PROT_READ, so a CPU store faults the process and a
 * GPU store faults the device context.  Consumers must treat the tensor as immutable. */
#ifndef WT_DLPACK_H_
#define WT_DLPACK_H_

#include <stdint.h>

#include "wt.h"

#ifdef __cplusplus
extern "C" {
#endif

/* ---- DLPack ABI (subset used here; layout as published) ---- */
#ifndef DLPACK_MAJOR_VERSION
typedef struct {
  uint32_t major;
  uint32_t minor;
} DLPackVersion;

typedef enum {
  kDLCPU = 1,
  kDLCUDA = 2,
  kDLCUDAHost = 3,
} DLDeviceType;

typedef struct {
  DLDeviceType device_type;
  int32_t device_id;
} DLDevice;

typedef enum {
  kDLInt = 0U,
  kDLUInt = 1U,
  kDLFloat = 2U,
  kDLBfloat = 4U,
} DLDataTypeCode;

typedef struct {
  uint8_t code;
  uint8_t bits;
  uint16_t lanes;
} DLDataType;

typedef struct {
  void *data;
  DLDevice device;
  int32_t ndim;
  DLDataType dtype;
  int64_t *shape;
  int64_t *strides;
  uint64_t byte_offset;
} DLTensor;

typedef struct DLManagedTensorVersioned {
  DLPackVersion version;
  void *manager_ctx;
  void (*deleter)(struct DLManagedTensorVersioned *self);
  uint64_t flags;
  DLTensor dl_tensor;
} DLManagedTensorVersioned;

#define DLPACK_FLAG_BITMASK_READ_ONLY (1ULL << 0)
#endif

/* Producer flags. */
#define WT_DLPACK_DEVICE 0u    /* kDLCUDA on the current device: the GPU reads the mapped pages
                                * in place (through the host page tables where the device
                                * supports it, else through a mapped host registration) */
#define WT_DLPACK_HOST (1u << 0) /* kDLCPU: a host tensor over the mapped pages (no CUDA call) */

/* Algorithm 1: one page-aligned tensor file of shape (M, K) and dtype `dtype` (WT_F32 ...
 * WT_U8).  Reject (WT_EINVAL) unless the file's size n equals M*K*sizeof(dtype) and n is a
 * non-zero multiple of the page size (a partial last page would alias whatever follows).
 * mmap(n, PROT_READ, MAP_SHARED), close the descriptor, expose the range (flags above), and
 * return a capsule with shape (M, K), explicit strides (K, 1), byte_offset 0, version 1.0
 * and the read-only flag.  Errors: WT_EINVAL, WT_EIO (open/fstat/mmap; errno in the
 * message), WT_ENOTSUP (no device route to host pages), WT_ENOMEM, WT_ECUDA. */
int wt_dlpack_file(const char *path, int32_t dtype, uint64_t M, uint64_t K, unsigned flags,
                   DLManagedTensorVersioned **out);

/* Tensor i of an open handle as its own capsule: its own read-only shared mapping of the
 * pages that hold the tensor (the data pointer sits at the tensor's offset inside the first
 * page), the tensor's own shape with compact strides, independent of the handle's lifetime
 * (wt_close does not invalidate it).  Zero-byte tensors are rejected (WT_EINVAL).  The pages
 * at the two ends may hold neighbouring tensors' bytes; they are read-only.  Errors as
 * wt_dlpack_file, plus WT_EINVAL for a bad index or a host-only handle with flags 0. */
int wt_dlpack_tensor(const wt_handle *h, size_t i, unsigned flags, DLManagedTensorVersioned **out);

/* Calls t->deleter(t) (for owners that never hand the capsule to a consumer).  NULL is a no-op. */
void wt_dlpack_release(DLManagedTensorVersioned *t);

/* Capsules produced and not yet deleted, process-wide (leak checks). */
int wt_dlpack_live(int64_t *n);

#ifdef __cplusplus
}
#endif

#endif /* WT_DLPACK_H_ */
