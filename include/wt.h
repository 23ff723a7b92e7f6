/*
 * wt — file-backed weights into GB300 device tensors, and the bandwidth-bound
 * consumer pass over them.  C ABI.
 *
 * The problem this library solves is the one the paper calls the ingestion
 * tax (Sec. 1; Sec. 2.2): checkpoint bytes that already sit in the page cache
 * must become ordinary device tensors that a kernel in the caller's stream
 * consumes.  The calls follow the paper's producer and execution contract:
 *
 *   wt_open   guarded open + shared read-only map of each file (Algorithm 1:
 *             size guard, mmap(PROT_READ, MAP_SHARED), close the descriptor)
 *             and the device-access route for the mapping (Sec. 7.3: registration
 *             and direct read are probed separately).
 *   wt_adopt  moves tensor bytes into caller-owned device memory and returns a
 *             per-tensor ready event (contract C3: order on the GPU).
 *   wt_pass   one GEMV per matrix in the caller's stream, each launch gated
 *             by its tensors' events, outputs kept on the device (C2).
 *   wt_checksum / wt_checksum_plain  per-tensor FNV-1a-64 digests of device
 *             bytes (the checksums of Sec. 6.1 that confirm kernels read the
 *             intended bytes).
 *   wt_close  waits for the library's own work on the mappings, unregisters,
 *             unmaps (Algorithm 1's deleter; Sec. 5.1 lifetime rules).
 *
 * Conventions
 *   - Every call returns int: WT_OK (0) or a negative WT_E* code.  No C++
 *     exception crosses this boundary.  wt_last_error() returns a thread-local
 *     message for the last failing call on the calling thread.
 *   - Streams and events are CUDA handles passed as void* (cudaStream_t,
 *     cudaEvent_t); a NULL stream is the legacy default stream.
 *   - Device pointers are caller-owned (the library never frees them).  The
 *     library borrows a destination until the event it returned completes.
 *   - The library never writes to a mapping.  A destination that lies inside
 *     one of the handle's mappings is rejected with WT_EINVAL (Sec. 5.1:
 *     read-only intent must be enforced before dispatch).
 *   - All kernels run on the device that is current when wt_open is called.
 */
#ifndef WT_H_
#define WT_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes -------------------------------------------------------- */
#define WT_OK 0
#define WT_EINVAL (-1)    /* bad argument (null, size, alignment, index, dtype) */
#define WT_EIO (-2)       /* open/read/mmap failed; errno in the message */
#define WT_EFORMAT (-3)   /* file violates the container format; file, entry, reason in the message */
#define WT_ENOMEM (-4)    /* host or device allocation failed */
#define WT_ECUDA (-5)     /* a CUDA runtime call failed; its error string in the message */
#define WT_ENOTSUP (-6)   /* route or dtype not available on this device/handle */
#define WT_ETIMEDOUT (-7) /* a bounded device wait gave up (see wt_device_status) */

/* ---- element types (the container's dtype byte) -------------------------- */
#define WT_F32 0
#define WT_BF16 1
#define WT_F16 2
#define WT_I8 3
#define WT_U8 4

/* ---- wt_open flags --------------------------------------------------------
 * Route for device reads of the mapping (one of the first four; default AUTO):
 *   AUTO       direct read when the device reads pageable memory through the
 *              host page tables (Grace ATS), else cudaHostRegister, else NONE.
 *   REGISTER   cudaHostRegister(Mapped) each whole-file mapping (ReadOnly is
 *              tried first and dropped if the driver rejects it).
 *   DIRECT     device reads the pageable mapping in place (no registration).
 *   NONE       the device never touches the mapping; only WT_ADOPT_STAGED works.
 * HOST_ONLY    parse and map only; no CUDA call at all (index inspection).
 * PREFAULT     populate every mapping's page-table entries at open
 *              (MADV_POPULATE_READ); otherwise wt_adopt populates each batch's
 *              source range just before it enqueues that batch.
 * NOMAP        parse and validate each file (open, fstat, pread of the index, close)
 *              but map nothing: the route of every file is NONE, tensor host_ptr is
 *              NULL, and only WT_ADOPT_STAGED adopts, reading the bytes with pread
 *              into the pinned ring (after checking that each path still names the
 *              file that was parsed: device, inode, size, mtime; WT_EIO otherwise).
 *              For checkpoints of many small files, where mapping every file costs
 *              more host time than their bytes take on the link (Sec. 5.3: the
 *              2506-file spine's map cost).  Not with REGISTER, DIRECT or PREFAULT.
 * MAP_LARGE    map only the files of at least WT_MAP_MIN_BYTES (the environment variable
 *              WT_MAP_MIN_BYTES, in bytes, overrides it); parse the smaller ones as NOMAP
 *              does (no mapping, route NONE, host_ptr NULL).  wt_adopt in GATHER or CE
 *              mode then moves the tensors of those small files as STAGED does (pread on
 *              host threads into the pinned ring, gather from the slot).  It does so on an
 *              internal stream, ordered after `stream`'s earlier work and concurrent with
 *              the mapped files' transfer, and `stream` waits for it before wt_adopt
 *              returns.  Each mapping costs an mmap and a page-table population, both
 *              serialised on the process's address-space lock, while a pread costs host
 *              copy bandwidth only.  So a checkpoint of many small files (Sec. 5.3)
 *              splits its host cost over both.  Not with NOMAP; PREFAULT covers the mapped
 *              files only.
 * TIMELINE     record a timing event before and after every ingest batch of
 *              wt_adopt and every GEMV group of wt_pass (outside stream capture),
 *              for wt_trace: the per-tensor overlap timeline of the first use.
 *              The ready events wt_adopt returns then carry timing too.
 * STAMPS       every one-column resident GEMV launch of wt_pass on the handle runs the
 *              stamping instantiation of its kernel, which also writes per-CTA
 *              %globaltimer stamps (the WT_STAMP_* record below) for wt_pass_stamps:
 *              where a small pass spends its time (prologue, plan-table reads, first
 *              copy, streaming, tail).  Same results; a diagnostic, not for timing runs.
 */
#define WT_ROUTE_AUTO 0u
#define WT_ROUTE_REGISTER 1u
#define WT_ROUTE_DIRECT 2u
#define WT_ROUTE_NONE 3u
#define WT_ROUTE_MASK 3u
#define WT_OPEN_HOST_ONLY (1u << 4)
#define WT_OPEN_PREFAULT (1u << 5)
#define WT_OPEN_TIMELINE (1u << 6)  /* timing events around every ingest batch and GEMV group (wt_trace) */
#define WT_OPEN_NOMAP (1u << 7)     /* parse only; no mapping; staged adopt reads with pread */
#define WT_OPEN_STAMPS (1u << 8)    /* per-CTA stamps of each one-column GEMV launch (wt_pass_stamps) */
#define WT_OPEN_MAP_LARGE (1u << 9) /* map files of >= WT_MAP_MIN_BYTES only; adopt the rest via pread */
#define WT_MAP_MIN_BYTES (1u << 18) /* WT_OPEN_MAP_LARGE's default threshold (file size, bytes) */

/* ---- wt_adopt modes ---------------------------------------------------------
 *   GATHER   SM gather kernel: 16-byte vector loads from the device-readable
 *            mapping, coalesced stores to HBM (the default).
 *   CE       copy engine: cudaMemcpyAsync from the device-readable mapping.
 *   STAGED   host threads copy page-cache bytes into a pinned ring (memcpy from
 *            the mapping, or pread for WT_OPEN_NOMAP files) and the gather kernel
 *            moves each slot to its destinations over the host link (the paper's
 *            staged/overlapped copy arm, Table "tab:tax" and Table
 *            "tab:gh-endpoints").  The ring (4 x 64 MiB of pinned memory per
 *            device) is allocated by the first staged adopt on a device and kept
 *            until the process exits; staged adopts on one device take turns on it.
 */
#define WT_ADOPT_GATHER 0u
#define WT_ADOPT_CE 1u
#define WT_ADOPT_STAGED 2u

typedef struct wt_handle wt_handle;

typedef struct {
  const char *name;     /* NUL-terminated, valid until wt_close */
  int32_t dtype;        /* WT_F32 ... WT_U8 */
  int32_t ndim;         /* 1..4 */
  uint64_t shape[4];    /* unused dims are 0 */
  uint64_t nbytes;      /* prod(shape) * sizeof(dtype) */
  uint32_t file;        /* index into the wt_open path list */
  uint64_t offset;      /* absolute file offset, multiple of 64 */
  const void *host_ptr; /* address of the blob in the read-only mapping (NULL: WT_OPEN_NOMAP) */
} wt_tensor_meta;

/* One GEMV of wt_pass: y[M] = W[M,K] . x[K], fp32 accumulate (Sec. 3.1 protocol:
 * one single-token GEMV per matrix).  W is row-major [out, in]; y is fp32.  For WT_F32,
 * WT_BF16 and WT_F16 weights x has W's dtype and scale is NULL.  For WT_I8 weights (the
 * paper's packed-int8 kernel with fp16 row scales, Sec. 3.1 and Table "tab:tax") x is
 * fp16 and scale points at M fp16 row scales: y_i = scale_i * sum_j W_ij x_j.  All
 * pointers are caller-owned device memory (or, for W, the handle's mapping: see
 * wt_pass).  wait_event (a cudaEvent_t from wt_adopt, or NULL) gates this GEMV on the GPU.
 *
 * cols = T in 1..16 selects the multi-column kernel (the paper's multi-column packed-int8
 * GEMV of the T-sweep, Sec. 4.3; each weight read serves all T activation columns):
 * x is X[T, K] row-major (column t = activation vector t, row pitch K elements) and y is
 * Y[T, M] row-major fp32, Y[t] = diag(scale) W X[t].  It runs on the tensor cores (fp16 or
 * bf16 products, fp32 accumulate) for WT_BF16, WT_F16 and WT_I8 weights; WT_F32 weights
 * with cols > 0 are WT_ENOTSUP.  cols = 0 is the one-column GEMV above. */
typedef struct {
  const void *W;
  int32_t dtype;        /* WT_F32, WT_BF16, WT_F16 or WT_I8 */
  int32_t cols;         /* 0: y = W x; 1..16: Y[T, M] from X[T, K] (see above) */
  uint64_t M;
  uint64_t K;
  const void *x;
  float *y;
  void *wait_event;
  const void *scale;    /* WT_I8: fp16 [M] row scales; otherwise NULL */
} wt_gemv_desc;

/* Thread-local message describing the last failure on this thread ("" if none). */
const char *wt_last_error(void);

/* ABI version of this header (increments on any incompatible change). */
int wt_abi_version(void);

/* Open n_paths checkpoint files (n_paths may be 0: a context for wt_pass and
 * wt_checksum only).  Per file: open(O_RDONLY), fstat, pread the header and the
 * length-prefixed index, validate every entry (dtype, ndim 1..4, nbytes ==
 * prod(shape)*sizeof(dtype) without overflow, offset % 64 == 0, blob after the
 * index, inside the file, in index order, no overlap, unique non-empty names,
 * index length exactly consumed), mmap(PROT_READ, MAP_SHARED), close the fd,
 * then set up the route.  On any failure nothing stays open or mapped and
 * *out is NULL.  Errors: WT_EINVAL, WT_EIO, WT_EFORMAT, WT_ENOMEM, WT_ECUDA,
 * WT_ENOTSUP (route requested but unavailable). */
int wt_open(const char *const *paths, int n_paths, unsigned flags, wt_handle **out);

int wt_num_tensors(const wt_handle *h, size_t *n);
int wt_num_files(const wt_handle *h, size_t *n);
/* Tensor i in (file, index) order. */
int wt_tensor_info(const wt_handle *h, size_t i, wt_tensor_meta *out);
/* wt_tensor_info of tensors [first, first + n) into out[0..n), in one call (a checkpoint of
 * thousands of files has thousands of entries).  Errors: WT_EINVAL (range, NULL). */
int wt_tensor_table(const wt_handle *h, size_t first, size_t n, wt_tensor_meta *out);
/* Every tensor name, in tensor order, each followed by a NUL byte, into buf.  *needed receives
 * the bytes required; with cap == 0 only *needed is set.  Errors: WT_EINVAL (NULL, cap too
 * small). */
int wt_tensor_names(const wt_handle *h, char *buf, size_t cap, size_t *needed);
/* Logical tensors of an open checkpoint.  A checkpoint may split a matrix's rows across
 * files (the paper's many-small spine, Sec. 5.3): a tensor named "<base>#r<k>", where k is
 * one to nine decimal digits, is row block k of the logical tensor <base>, and the blocks of
 * one base, from any file, form one logical tensor.  Every other tensor is a logical tensor
 * of its own.  group[i] receives the logical tensor of tensor i, numbered 0.. in order of
 * first appearance; block[i] receives k, or -1 for a tensor that is not a row block.  Both
 * arrays have wt_num_tensors entries (the caller's); *n_groups receives the number of
 * logical tensors.  Whether the blocks of a group stack (2-D, one dtype, one row length,
 * distinct k) is the caller's check.  Errors: WT_EINVAL (NULL). */
int wt_tensor_groups(const wt_handle *h, uint32_t *group, int32_t *block, size_t *n_groups);
/* First tensor whose name equals `name`; WT_EINVAL if none. */
int wt_find(const wt_handle *h, const char *name, size_t *i);
/* Route actually taken for file f (WT_ROUTE_REGISTER / DIRECT / NONE). */
int wt_file_route(const wt_handle *h, size_t f, unsigned *route);
/* The cudaHostRegister flags file f's registration holds: cudaHostRegisterMapped (0x02),
 * with cudaHostRegisterReadOnly (0x08) when the driver accepted read-only registration of
 * the file-backed pages, or 0 when the file is not registered (routes DIRECT and NONE).
 * The REGISTER route asks for read-only first and, when the driver refuses it, registers
 * the PROT_READ mapping without the flag; this call tells the two apart (Sec. 5.1: the
 * read-only intent is then enforced by the mapping's protection and the host-side checks,
 * not by the registration).  Errors: WT_EINVAL. */
int wt_file_registration(const wt_handle *h, size_t f, unsigned *flags);

/* Host time wt_open spent in each of the hot path's first three steps (Sec. 5.3's map-and-
 * wire cost, per phase), measured inside the call with a monotonic clock:
 *   index_ms      wall time of the parallel loop that opens, parses and validates every file
 *                 and maps those it maps (steps 1 and 2 together, on the host pool);
 *   index_cpu_ms  summed over the files: open, fstat, index reads and validation (step 1);
 *   map_cpu_ms    summed over the files: mmap (step 2; the calls serialise on the process's
 *                 address-space lock, so this is close to their wall time);
 *   prefault_ms   wall time of WT_OPEN_PREFAULT's population (0 without it);
 *   route_ms      wall time of the route probe and any registration (step 3);
 *   files_mapped, files_registered: how many files each step touched.
 * Errors: WT_EINVAL (NULL argument). */
typedef struct {
  double index_ms;
  double index_cpu_ms;
  double map_cpu_ms;
  double prefault_ms;
  double route_ms;
  uint64_t files_mapped;
  uint64_t files_registered;
} wt_open_phases;
int wt_open_times(const wt_handle *h, wt_open_phases *out);

/* Copy tensors idx[0..n) into device memory dst[0..n) (each at least nbytes of
 * that tensor, 16-byte aligned for the vector path) on `stream`, in order.
 * Tensors are grouped into batches of a few MB to a few hundred MB; one event
 * is recorded after each batch and ready[i] receives the event of tensor i's
 * batch (several entries may hold the same event).  Events are owned by the
 * handle and destroyed by wt_close.  Because the batches run in order on one
 * stream, ready[i] also implies every earlier tensor of this call.  STAGED
 * mode blocks the calling thread until every byte has left the page cache
 * (the copy engine may still be draining the last slots).
 * Errors: WT_EINVAL (index, null, overlap with a mapping, a dst that starts in a device
 * allocation and runs past its end), WT_ENOTSUP (mode needs a device route the file
 * lacks), WT_ENOMEM, WT_ECUDA. */
int wt_adopt(wt_handle *h, const size_t *idx, void *const *dst, size_t n, unsigned mode,
             void *stream, void **ready);

/* Enqueue one GEMV per descriptor on `stream`.  W may be device memory (the resident
 * endpoint: TMA-fed kernel streaming HBM) or lie inside one of this handle's file mappings
 * (the map endpoint of Sec. 8.1, contract C1: the kernel reads the mapped rows in place over
 * the host link, no copy; the rows are populated once when the plan is built and must stay
 * resident, Algorithm 2's precondition).  y must not lie inside a mapping.  Descriptors that
 * carry the same wait_event form one group, wherever they stand in the list (those with
 * none form one group too); groups are enqueued in order of their first descriptor.  For
 * each group the stream waits on its event (cudaStreamWaitEvent, never a host wait) and one
 * persistent launch streams every matrix of the group, rows split evenly across the SMs.  Repeated
 * calls with identical descriptors reuse a cached launch plan.  The result of
 * a row does not depend on how rows were grouped or split (deterministic, no
 * floating-point atomics).
 *
 * Stream capture: a wt_pass issued on a stream that is being captured into a CUDA graph
 * records the pass's launches into the graph (replays then cost no host work).  The same
 * descriptors must have run through wt_pass once before, outside the capture, and that
 * stream must have been synchronised since (the plan's tables must be in device memory);
 * otherwise the call returns WT_EINVAL before issuing any CUDA call.  The captured plan is
 * kept until wt_close; every replay must complete before wt_close.
 *
 * Errors: WT_EINVAL (null pointer with M*K > 0, cols outside 0..16, dimension > 2^31-1, a
 * capture without the warm-up call, an operand that starts in a device allocation and runs
 * past its end), WT_ENOTSUP (dtype), WT_ENOMEM, WT_ECUDA. */
int wt_pass(wt_handle *h, const wt_gemv_desc *d, size_t n, void *stream);

/* Leaf-tree FNV-1a-64 digest of each device buffer ptr[i] (nbytes[i] bytes),
 * written to out_dev[i] (device memory, caller-owned).  D_tree = FNV-1a-64 over
 * the 8-byte little-endian encodings of [nbytes, leaf_0, ..., leaf_{L-1}],
 * leaf_k = FNV-1a-64 of bytes [4096k, min(4096(k+1), nbytes)).  Temporary leaf
 * storage is stream-ordered (cudaMallocAsync/cudaFreeAsync on `stream`). */
int wt_checksum(wt_handle *h, const void *const *ptr, const uint64_t *nbytes, size_t n,
                uint64_t *out_dev, void *stream);

/* Literal FNV-1a-64 of each device buffer (one serial chain per buffer; meant
 * for verification).  Buffers above 256 MiB are rejected with WT_EINVAL. */
int wt_checksum_plain(wt_handle *h, const void *const *ptr, const uint64_t *nbytes, size_t n,
                      uint64_t *out_dev, void *stream);

/* Leaf-tree digests exactly as wt_checksum computes them, for callers that must
 * not allocate device memory: code inside an allocator hook (it would re-enter
 * the allocator it serves), programs whose device memory is all handed to
 * their own pool, and loops that cannot take the device-wide synchronisation
 * of cudaFree.  The paper has no counterpart; this is a library convenience.
 * No handle is needed.  The leaf digests and the chunk tables of the parallel
 * second level live in an array of about 8.7 MiB compiled into the library
 * (every GPU that loads the library keeps it until exit); a call
 * whose buffers need more than 1,048,576 leaves of 4096 bytes (4 GiB of input
 * in total) is rejected with WT_EINVAL, before any CUDA call.  The first call on each device
 * looks up that array's device address (cudaGetSymbolAddress) with the device
 * current and remembers it with the CUDA context that was current; make that first call
 * before any stream capture.  Under another context (after cudaDeviceReset, or a context
 * created through the driver API) the array is a different one and the address is looked
 * up again, so such a first call, too, belongs outside a capture.  Calls share the
 * array, so two calls whose kernels overlap on the GPU race; calls ordered on
 * one stream do not.  Nothing in the array needs clearing between calls.
 * Errors: WT_EINVAL (NULL array or buffer, too large), WT_ECUDA. */
int wt_checksum_noalloc(const void *const *ptr, const uint64_t *nbytes, size_t n, uint64_t *out_dev,
                        void *stream);

/* One record of the first-use timeline (handles opened with WT_OPEN_TIMELINE).  An ingest
 * record is one batch of wt_adopt: begin when its stream reached the batch, end when its
 * bytes had landed (the ready event of its tensors).  A GEMV record is one group of wt_pass:
 * begin when its stream had waited for the group's event and reached its first launch, end
 * when its last launch had finished.  Contract C3 (Table "tab:contract"; Sec. 4.3) holds
 * when each group begins right after its batch ends, not after the last batch. */
#define WT_TRACE_INGEST 0
#define WT_TRACE_GEMV 1
typedef struct {
  int32_t kind;      /* WT_TRACE_INGEST or WT_TRACE_GEMV */
  int32_t pad;
  uint64_t index;    /* ordinal of the batch (or group) within the handle, in enqueue order */
  uint64_t bytes;    /* bytes the batch moved, or weight bytes the group's GEMVs stream */
  void *event;       /* ingest: the batch's ready event, as wt_adopt returned it for the
                        tensors whose last byte the batch holds; GEMV: the wait_event of the
                        group's descriptors (NULL: none) */
  double begin_ms;   /* milliseconds from the origin event */
  double end_ms;
} wt_trace_rec;

/* Read the handle's timeline: waits for every recorded event, writes the first min(cap, *n)
 * records (in enqueue order, ingest batches and GEMV groups interleaved as they were
 * enqueued) with times relative to `origin` (a cudaEvent_t created with timing and recorded
 * before the traced work, e.g. on the ingest stream just before wt_adopt), sets *n to the
 * number recorded, then releases them (a second call returns only later records).  Blocks
 * the calling thread.  Errors: WT_EINVAL (NULL argument, handle without WT_OPEN_TIMELINE),
 * WT_ECUDA (e.g. origin without timing, or not recorded). */
int wt_trace(wt_handle *h, void *origin, wt_trace_rec *out, size_t cap, size_t *n);

/* Per-CTA stamps of the latest one-column resident GEMV launch that wt_pass issued on a
 * handle opened with WT_OPEN_STAMPS (the persistent TMA kernel of Sec. 4.2's resident
 * consumer; the multi-column, map-endpoint and split-K reduction kernels are not stamped).
 * Each CTA has WT_STAMP_FIELDS words, CTA b at out[b * WT_STAMP_FIELDS]; every field but
 * WT_STAMP_SM is the GPU's global nanosecond timer (comparable across SMs), and a field
 * the CTA never reached (a CTA with no rows) is 0.  "Latest" is in host issue order: for a
 * pass captured in a CUDA graph, the stamps of its latest replay.  Waits until the device
 * is idle, copies min(cap, *n) CTAs' records to out (host memory) and sets *n to the
 * launch's grid (0: no stamped launch yet).  Errors: WT_EINVAL (NULL argument, handle
 * without WT_OPEN_STAMPS), WT_ECUDA. */
#define WT_STAMP_ENTRY 0       /* CTA entry */
#define WT_STAMP_PROLOGUE 1    /* mbarriers initialised (shared-memory set-up done) */
#define WT_STAMP_OPERANDS 2    /* past the wait for the previous grid of the stream (a
                                  programmatic launch in a captured graph); operands readable */
#define WT_STAMP_FIRST_COPY 3  /* first bulk copy issued (after the plan-table reads) */
#define WT_STAMP_FIRST_FULL 4  /* first stage landed, as the first consumer warp saw it */
#define WT_STAMP_LAST_FULL 5   /* last stage landed, as the first consumer warp saw it */
#define WT_STAMP_EXIT 6        /* every warp of the CTA done */
#define WT_STAMP_SM 7          /* the SM the CTA ran on (not a time) */
#define WT_STAMP_FIELDS 8
int wt_pass_stamps(wt_handle *h, uint64_t *out, size_t cap, size_t *n);

/* Device-side status word of the handle: 0, or the first WT_ETIMEDOUT-class
 * code a bounded wait inside a kernel recorded (reads it synchronously). */
int wt_device_status(wt_handle *h, int *status);

/* Bytes of the handle's file mappings that are resident in the page cache right now
 * (mincore over every mapping, page granular, clipped to the file sizes) and their total
 * (WT_ENOTSUP for a WT_OPEN_NOMAP handle, which maps nothing).
 * Algorithm 2 stops with "storage-bound" when the mapped set is not resident (Sec. 8.1);
 * Table "controls" queries residency before and after a measurement.  Host-only handles
 * work too.  Errors: WT_EINVAL, WT_EIO. */
int wt_residency(const wt_handle *h, uint64_t *resident, uint64_t *total);

/* Kernels this handle has launched so far (gather, GEMV, checksum launches). */
int wt_kernel_launches(const wt_handle *h, uint64_t *n);

/* Objects the library holds right now, over all handles of the process: open handles,
 * cached launch plans, CUDA events it created, and the device and pinned host bytes it
 * allocated itself and has handed out (status words, plan tables, split-K workspaces, the
 * staged ring).  Buffers the caller owns are not counted.  After wt_close of every handle
 * these five return to their earlier values (Sec. 5.1: a producer's lifetime leaves nothing
 * behind; the 200-cycle checks read these), except that the first staged adopt on a device
 * adds its ring for good: 4 events and 268,435,456 pinned bytes.
 * cached_device_bytes and cached_pinned_bytes are the blocks a closed handle gave back and
 * the library keeps, per device, for the next handle (so that opening and using a handle
 * calls no cudaMalloc, cudaHostAlloc or cudaFree once the cache holds its sizes); they are
 * bounded by 256 MiB per device and kind and stay until the process exits.
 * Errors: WT_EINVAL. */
typedef struct {
  int64_t handles;
  int64_t plans;
  int64_t events;
  int64_t device_bytes;
  int64_t pinned_bytes;
  int64_t cached_device_bytes;
  int64_t cached_pinned_bytes;
} wt_live_counts;
int wt_live(wt_live_counts *out);

/* Wait for the library's own enqueued work that reads the mappings, then
 * cudaHostUnregister, munmap, destroy events, free library allocations.
 * NULL is a no-op.  Callable from any thread. */
int wt_close(wt_handle *h);

#ifdef __cplusplus
}
#endif

#endif /* WT_H_ */
