/* Plain CPU Allreduce by its definition: every rank ends with the op-reduction of all
 * P input vectors (Sec. "Introduction", MPI_Allreduce semantics), computed element by
 * element in rank order and written to every rank's output.
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only tests/ and the CPU-baseline leg of
 * bench.py load it: it is the multi-threaded CPU baseline beside the single-threaded
 * oracle, and a second, independent implementation of the definition that the oracle's
 * exact cases are checked against (int32 wraparound sums and max/min do not depend on
 * the association order).  It shares no code with the CUDA library.
 *
 * Element types: 0 = fp32 (the sum runs in double, rank order, and is rounded to fp32
 * once), 2 = int32 (two's-complement wraparound).  Ops: 0 = sum, 1 = max, 2 = min.
 * bf16 is not handled.  Threads split the element range into contiguous pieces;
 * threads <= 1 runs on the calling thread.  Returns 0, or -1 on a bad argument.
 */
#include <pthread.h>
#include <stddef.h>
#include <stdint.h>

typedef struct {
  const void *const *in;
  void *const *out;
  int P, dtype, op;
  size_t lo, hi;
} job_t;

/* Elements go in blocks of BLK: for every element the ranks are still combined in rank
 * order, but each rank's block is read contiguously, so the inner loops stream and
 * vectorise. */
enum { BLK = 512 };

static void reduce_f32(const job_t *j) {
  const float *const *in = (const float *const *)j->in;
  float *const *out = (float *const *)j->out;
  double acc[BLK];
  float r[BLK];
  for (size_t e0 = j->lo; e0 < j->hi; e0 += BLK) {
    const size_t m = (j->hi - e0) < BLK ? (j->hi - e0) : BLK;
    if (j->op == 0) {
      for (size_t k = 0; k < m; ++k) acc[k] = 0.0;
      for (int x = 0; x < j->P; ++x) {
        const float *v = in[x] + e0;
        for (size_t k = 0; k < m; ++k) acc[k] += (double)v[k];
      }
      for (size_t k = 0; k < m; ++k) r[k] = (float)acc[k];
    } else {
      for (size_t k = 0; k < m; ++k) r[k] = in[0][e0 + k];
      for (int x = 1; x < j->P; ++x) {
        const float *v = in[x] + e0;
        for (size_t k = 0; k < m; ++k)
          if (j->op == 1 ? v[k] > r[k] : v[k] < r[k]) r[k] = v[k];
      }
    }
    for (int x = 0; x < j->P; ++x) {
      float *o = out[x] + e0;
      for (size_t k = 0; k < m; ++k) o[k] = r[k];
    }
  }
}

static void reduce_i32(const job_t *j) {
  const int32_t *const *in = (const int32_t *const *)j->in;
  int32_t *const *out = (int32_t *const *)j->out;
  uint32_t acc[BLK];
  int32_t r[BLK];
  for (size_t e0 = j->lo; e0 < j->hi; e0 += BLK) {
    const size_t m = (j->hi - e0) < BLK ? (j->hi - e0) : BLK;
    if (j->op == 0) {
      for (size_t k = 0; k < m; ++k) acc[k] = 0u;
      for (int x = 0; x < j->P; ++x) {
        const int32_t *v = in[x] + e0;
        for (size_t k = 0; k < m; ++k) acc[k] += (uint32_t)v[k];
      }
      for (size_t k = 0; k < m; ++k) r[k] = (int32_t)acc[k];
    } else {
      for (size_t k = 0; k < m; ++k) r[k] = in[0][e0 + k];
      for (int x = 1; x < j->P; ++x) {
        const int32_t *v = in[x] + e0;
        for (size_t k = 0; k < m; ++k)
          if (j->op == 1 ? v[k] > r[k] : v[k] < r[k]) r[k] = v[k];
      }
    }
    for (int x = 0; x < j->P; ++x) {
      int32_t *o = out[x] + e0;
      for (size_t k = 0; k < m; ++k) o[k] = r[k];
    }
  }
}

static void *run(void *arg) {
  const job_t *j = (const job_t *)arg;
  if (j->dtype == 0)
    reduce_f32(j);
  else
    reduce_i32(j);
  return NULL;
}

int column_allreduce(const void *const *in, void *const *out, int P, size_t n, int dtype, int op,
                     int threads) {
  enum { MAX_THREADS = 256 };
  if (P < 1 || in == NULL || out == NULL || (dtype != 0 && dtype != 2) || op < 0 || op > 2)
    return -1;
  if (n == 0) return 0;
  if (threads < 1) threads = 1;
  if (threads > MAX_THREADS) threads = MAX_THREADS;
  if ((size_t)threads > n) threads = (int)n;
  job_t jobs[MAX_THREADS];
  pthread_t tid[MAX_THREADS];
  const size_t per = (n + (size_t)threads - 1) / (size_t)threads;
  for (int t = 0; t < threads; ++t) {
    jobs[t].in = in;
    jobs[t].out = out;
    jobs[t].P = P;
    jobs[t].dtype = dtype;
    jobs[t].op = op;
    jobs[t].lo = (size_t)t * per < n ? (size_t)t * per : n;
    jobs[t].hi = (size_t)(t + 1) * per < n ? (size_t)(t + 1) * per : n;
  }
  int started = 0;
  for (int t = 1; t < threads; ++t) {
    if (pthread_create(&tid[t], NULL, run, &jobs[t]) != 0) break;
    started = t;
  }
  run(&jobs[0]);
  for (int t = 1; t <= started; ++t) pthread_join(tid[t], NULL);
  /* pieces whose thread could not be started run here */
  for (int t = started + 1; t < threads; ++t) run(&jobs[t]);
  return 0;
}
