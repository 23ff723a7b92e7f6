/*
 * CPU oracle for the file-backed weight path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the bench's
 * CPU-baseline leg load this code.  It shares no code, header or table with
 * the CUDA library: it has its own file reader, its own index decoder, its own
 * checksums and its own GEMV.  It is plain, single-threaded and slow on
 * purpose, so that each function can be checked against its definition by eye.
 *
 *   O1  parse   read() the whole file into a heap buffer; decode the
 *               length-prefixed index byte by byte; apply the producer's
 *               guards (Algorithm 1: size = M*K*sizeof(dtype); Sec. 5.3:
 *               aligned bases) generalised to the container.
 *   O2  bytes   FNV-1a-64 of every blob (D_plain) and the leaf-tree digest
 *               (D_tree, 4096-byte leaves) defined below.
 *   O3  GEMV    y_i = sum_j W_ij x_j in fp64, in index order, plus
 *               a_i = sum_j |W_ij x_j| (the per-row error normaliser).  The
 *               consumer pass the paper times over adopted storage (Sec. 3.1,
 *               Table "tab:tax"; one GEMV per matrix).
 *
 * Readings (the paper leaves these open):
 *   - "per-tensor 64-bit FNV-1a": D_plain is the literal FNV-1a-64 of the
 *     blob.  D_tree is FNV-1a-64 over the 8-byte little-endian encodings of
 *     [nbytes, leaf_0, ..., leaf_{L-1}], leaf_k = D_plain of bytes
 *     [4096k, min(4096(k+1), n)), L = ceil(n/4096) (no leaves when n = 0).
 *   - bf16 decodes as (u16 << 16) reinterpreted as an IEEE single; f16 is
 *     decoded from its sign/exponent/mantissa fields; both widen exactly.
 *
 * Pins (tests/test_oracle_*.py): the FNV offset basis re-derived from the FNV
 * specification's own construction; step-by-step inversion of the hash with
 * the prime's modular inverse; D_tree/D_plain tie for n <= 4096; brute-force
 * GEMV on integer-valued matrices; one-hot x giving exact columns; x = 1
 * giving row sums; an index round trip and every rejection rule on
 * hand-built files.
 */
#include <errno.h>
#include <fcntl.h>
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <sys/stat.h>
#include <unistd.h>

#define OR_FNV_OFFSET 0xcbf29ce484222325ULL
#define OR_FNV_PRIME 0x00000100000001b3ULL
#define OR_LEAF 4096ULL
#define OR_ALIGN 64ULL

typedef struct {
  char *name;
  int dtype;
  int ndim;
  uint64_t shape[4];
  uint64_t offset;
  uint64_t nbytes;
} or_entry;

typedef struct {
  uint8_t *bytes;
  uint64_t size;
  uint64_t index_bytes;
  uint32_t n;
  or_entry *e;
} or_file;

static char or_err[512];

const char *or_last_error(void) { return or_err; }

static uint64_t rd_le(const uint8_t *p, int nbytes) {
  uint64_t v = 0;
  for (int i = nbytes - 1; i >= 0; --i) v = (v << 8) | p[i];
  return v;
}

static int elem_size(int dtype) {
  switch (dtype) {
    case 0: return 4; /* f32 */
    case 1: return 2; /* bf16 */
    case 2: return 2; /* f16 */
    case 3: return 1; /* i8 */
    case 4: return 1; /* u8 */
    default: return 0;
  }
}

void or_free(or_file *f) {
  if (!f) return;
  if (f->e) {
    for (uint32_t i = 0; i < f->n; ++i) free(f->e[i].name);
    free(f->e);
  }
  free(f->bytes);
  free(f);
}

static int fail(or_file *f, const char *path, const char *why, long long entry) {
  if (entry >= 0)
    snprintf(or_err, sizeof or_err, "%s: entry %lld: %s", path, entry, why);
  else
    snprintf(or_err, sizeof or_err, "%s: %s", path, why);
  or_free(f);
  return -1;
}

/* O1: read the whole file and decode + validate its index. */
int or_load(const char *path, or_file **out) {
  *out = NULL;
  or_file *f = (or_file *)calloc(1, sizeof *f);
  if (!f) return fail(NULL, path, "out of memory", -1);
  int fd = open(path, O_RDONLY);
  if (fd < 0) {
    snprintf(or_err, sizeof or_err, "%s: open: %s", path, strerror(errno));
    free(f);
    return -2;
  }
  struct stat st;
  if (fstat(fd, &st) != 0) {
    close(fd);
    return fail(f, path, "fstat failed", -1);
  }
  f->size = (uint64_t)st.st_size;
  f->bytes = (uint8_t *)malloc(f->size ? f->size : 1);
  if (!f->bytes) {
    close(fd);
    return fail(f, path, "out of memory", -1);
  }
  uint64_t got = 0;
  while (got < f->size) {
    ssize_t r = read(fd, f->bytes + got, f->size - got);
    if (r <= 0) {
      close(fd);
      return fail(f, path, "short read", -1);
    }
    got += (uint64_t)r;
  }
  close(fd);

  const uint8_t *b = f->bytes;
  if (f->size < 16) return fail(f, path, "file shorter than the 16-byte header", -1);
  if (memcmp(b, "WTCKPT01", 8) != 0) return fail(f, path, "bad magic", -1);
  f->index_bytes = rd_le(b + 8, 8);
  if (f->index_bytes < 4 || f->index_bytes > f->size - 16)
    return fail(f, path, "index length outside the file", -1);
  const uint8_t *ix = b + 16;
  const uint64_t ixn = f->index_bytes;
  uint64_t pos = 0;
  uint32_t n = (uint32_t)rd_le(ix, 4);
  pos = 4;
  /* every entry needs at least 2+1+1+1+8+8+8 = 29 bytes */
  if ((uint64_t)n * 29ULL > ixn - 4) return fail(f, path, "entry count exceeds the index", -1);
  f->e = (or_entry *)calloc(n ? n : 1, sizeof(or_entry));
  if (!f->e) return fail(f, path, "out of memory", -1);
  f->n = n;
  const uint64_t data_start = 16 + ixn;
  uint64_t prev_end = data_start;
  for (uint32_t i = 0; i < n; ++i) {
    or_entry *e = &f->e[i];
    if (pos + 2 > ixn) return fail(f, path, "index truncated (name length)", i);
    uint64_t nl = rd_le(ix + pos, 2);
    pos += 2;
    if (nl == 0) return fail(f, path, "empty name", i);
    if (pos + nl + 2 > ixn) return fail(f, path, "index truncated (name)", i);
    e->name = (char *)malloc(nl + 1);
    if (!e->name) return fail(f, path, "out of memory", i);
    for (uint64_t c = 0; c < nl; ++c) {
      if (ix[pos + c] == 0) return fail(f, path, "NUL byte in name", i);
      e->name[c] = (char)ix[pos + c];
    }
    e->name[nl] = 0;
    pos += nl;
    e->dtype = ix[pos];
    e->ndim = ix[pos + 1];
    pos += 2;
    if (elem_size(e->dtype) == 0) return fail(f, path, "unknown dtype", i);
    if (e->ndim < 1 || e->ndim > 4) return fail(f, path, "ndim outside 1..4", i);
    if (pos + 8ULL * (uint64_t)e->ndim + 16 > ixn) return fail(f, path, "index truncated (shape)", i);
    /* count = prod(shape) * sizeof(dtype), refusing any overflow */
    uint64_t count = (uint64_t)elem_size(e->dtype);
    int zero = 0;
    for (int d = 0; d < e->ndim; ++d) {
      e->shape[d] = rd_le(ix + pos, 8);
      pos += 8;
      if (e->shape[d] == 0) zero = 1;
    }
    if (!zero) {
      for (int d = 0; d < e->ndim; ++d) {
        if (count > UINT64_MAX / e->shape[d]) return fail(f, path, "shape product overflows", i);
        count *= e->shape[d];
      }
    } else {
      count = 0;
    }
    e->offset = rd_le(ix + pos, 8);
    e->nbytes = rd_le(ix + pos + 8, 8);
    pos += 16;
    /* Algorithm 1's size guard: the blob holds exactly prod(shape) elements */
    if (e->nbytes != count) return fail(f, path, "nbytes != prod(shape) * sizeof(dtype)", i);
    /* aligned base (Sec. 5.3), after the index, inside the file */
    if (e->offset % OR_ALIGN != 0) return fail(f, path, "offset not 64-byte aligned", i);
    if (e->offset < data_start) return fail(f, path, "blob overlaps the header or index", i);
    if (e->offset > f->size || e->nbytes > f->size - e->offset)
      return fail(f, path, "blob runs past the end of the file", i);
    /* blobs are stored in index order and do not overlap */
    if (e->offset < prev_end) return fail(f, path, "blob overlaps the previous blob", i);
    prev_end = e->offset + e->nbytes;
    for (uint32_t j = 0; j < i; ++j)
      if (strcmp(f->e[j].name, e->name) == 0) return fail(f, path, "duplicate name", i);
  }
  if (pos != ixn) return fail(f, path, "index length does not match its entries", -1);
  *out = f;
  return 0;
}

uint32_t or_count(const or_file *f) { return f->n; }
uint64_t or_size(const or_file *f) { return f->size; }
const uint8_t *or_bytes(const or_file *f) { return f->bytes; }

int or_entry_info(const or_file *f, uint32_t i, const char **name, int *dtype, int *ndim,
                  uint64_t *shape4, uint64_t *offset, uint64_t *nbytes) {
  if (i >= f->n) return -1;
  const or_entry *e = &f->e[i];
  *name = e->name;
  *dtype = e->dtype;
  *ndim = e->ndim;
  for (int d = 0; d < 4; ++d) shape4[d] = d < e->ndim ? e->shape[d] : 0;
  *offset = e->offset;
  *nbytes = e->nbytes;
  return 0;
}

/* O2: FNV-1a-64, one byte at a time: h ^= byte, then h *= prime (mod 2^64). */
uint64_t or_fnv1a64(const uint8_t *p, uint64_t n) {
  uint64_t h = OR_FNV_OFFSET;
  for (uint64_t i = 0; i < n; ++i) {
    h ^= (uint64_t)p[i];
    h *= OR_FNV_PRIME;
  }
  return h;
}

static uint64_t fnv_feed_le64(uint64_t h, uint64_t v) {
  for (int k = 0; k < 8; ++k) {
    h ^= (v >> (8 * k)) & 0xffULL;
    h *= OR_FNV_PRIME;
  }
  return h;
}

/* O2: leaf-tree digest.  FNV-1a-64 over LE64(n), LE64(leaf_0), ..., LE64(leaf_{L-1}). */
uint64_t or_fnv_tree(const uint8_t *p, uint64_t n) {
  uint64_t h = fnv_feed_le64(OR_FNV_OFFSET, n);
  for (uint64_t s = 0; s < n; s += OR_LEAF) {
    uint64_t len = n - s < OR_LEAF ? n - s : OR_LEAF;
    h = fnv_feed_le64(h, or_fnv1a64(p + s, len));
  }
  return h;
}

/* Decode one element of W or x to double (exact widening). */
static double f16_to_double(uint32_t h) {
  int s = (h >> 15) & 1;
  int e = (h >> 10) & 0x1f;
  uint32_t m = h & 0x3ff;
  double v;
  if (e == 0)
    v = ldexp((double)m, -24); /* subnormal: m * 2^-24 */
  else if (e == 31)
    v = m ? NAN : INFINITY;
  else
    v = ldexp((double)(m | 0x400), e - 25); /* (1024 + m) * 2^(e-15-10) */
  return s ? -v : v;
}

static double elem(const uint8_t *p, int dtype, uint64_t i) {
  if (dtype == 0) {
    uint32_t u = (uint32_t)rd_le(p + 4 * i, 4);
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
  }
  if (dtype == 1) {
    uint32_t u = (uint32_t)rd_le(p + 2 * i, 2) << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
  }
  if (dtype == 2) return f16_to_double((uint32_t)rd_le(p + 2 * i, 2));
  if (dtype == 3) return (double)(int8_t)p[i];
  return (double)p[i];
}

/* O3: one row.  yhat = sum_j W_rj x_j and a = sum_j |W_rj x_j|, fp64, j in index order. */
static void gemv_row(const uint8_t *W, int dtype, uint64_t K, const uint8_t *x, uint64_t r,
                     double *yhat, double *a) {
  const uint8_t *row = W + r * K * (uint64_t)elem_size(dtype);
  double s = 0.0, t = 0.0;
  for (uint64_t j = 0; j < K; ++j) {
    double p = elem(row, dtype, j) * elem(x, dtype, j);
    s += p;
    t += fabs(p);
  }
  *yhat = s;
  *a = t;
}

/* O3 over all M rows.  W is [M, K] row-major ([out, in]); x has W's dtype. */
int or_gemv(const uint8_t *W, int dtype, uint64_t M, uint64_t K, const uint8_t *x, double *yhat,
            double *a) {
  if (elem_size(dtype) == 0) return -1;
  for (uint64_t r = 0; r < M; ++r) gemv_row(W, dtype, K, x, r, &yhat[r], &a[r]);
  return 0;
}

/* O3 for int8 weights with fp16 row scales (the paper's single-token kernel, Sec. 3.1 and
 * Table "tab:tax"): yhat_i = s_i * sum_j W_ij x_j and a_i = |s_i| * sum_j |W_ij x_j| in fp64,
 * j in index order; W is int8 [M, K], s is fp16 [M], x is fp16 [K]. */
int or_gemv_q8(const uint8_t *W, const uint8_t *s, uint64_t M, uint64_t K, const uint8_t *x,
               const uint64_t *rows, uint64_t nrows, double *yhat, double *a) {
  for (uint64_t i = 0; i < nrows; ++i) {
    const uint64_t r = rows ? rows[i] : i;
    if (r >= M) return -1;
    const uint8_t *row = W + r * K;
    double acc = 0.0, abs_acc = 0.0;
    for (uint64_t j = 0; j < K; ++j) {
      const double p = (double)(int8_t)row[j] * elem(x, 2, j);
      acc += p;
      abs_acc += fabs(p);
    }
    const double sc = elem(s, 2, r);
    yhat[i] = sc * acc;
    a[i] = fabs(sc) * abs_acc;
  }
  return 0;
}

/* O3 for a chosen set of rows (full-size checks sample rows). */
int or_gemv_rows(const uint8_t *W, int dtype, uint64_t M, uint64_t K, const uint8_t *x,
                 const uint64_t *rows, uint64_t nrows, double *yhat, double *a) {
  if (elem_size(dtype) == 0) return -1;
  for (uint64_t i = 0; i < nrows; ++i) {
    if (rows[i] >= M) return -1;
    gemv_row(W, dtype, K, x, rows[i], &yhat[i], &a[i]);
  }
  return 0;
}
