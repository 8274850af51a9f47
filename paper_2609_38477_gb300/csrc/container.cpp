// Container file of a compressed model: the global decoder table (Sec. 3.6:
// hull rungs, thresholds, tied threshold, floor) and, per tensor, what Alg. 2
// reads besides the table: shape, the importance factors a and rho (the
// decoder recomputes the rung map from them), the tie count T_t, the FP16
// outlier columns (Sec. 3.5) and the payload bit stream.  Host code only.
//
// Layout (all little-endian, no padding):
//   "SEEDQ\0v1"                       8 bytes
//   u32 version (1), u32 J
//   J x (i32 S, i32 k); (J-1) x f64 theta; i32 j_tie; f64 q
//   9 x u32 LFSR taps for S = 8..16 (the stream's generator; must match)
//   u32 ntensors
//   per tensor: u32 name_len, name bytes; i64 R; i64 C; f32 a[C];
//               u32 has_rho, f32 rho[R] if has_rho; i64 tie_count;
//               i32 n_out, i32 cols[n_out], u16 vals[R * n_out];
//               u64 stream_bits, u64 stream_len = ceil(bits / 8), stream bytes
//   u64 FNV-1a hash of every preceding byte
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <new>
#include <string>
#include <vector>

#include "../../include/seedq.h"

namespace {

const char kMagic[8] = {'S', 'E', 'E', 'D', 'Q', '\0', 'v', '1'};

uint64_t fnv1a(const uint8_t *p, size_t n) {
  uint64_t h = 0xcbf29ce484222325ull;
  for (size_t i = 0; i < n; ++i) {
    h ^= p[i];
    h *= 0x100000001b3ull;
  }
  return h;
}

// Little-endian encoding independent of the host's byte order.
struct Writer {
  std::vector<uint8_t> buf;
  void bytes(const void *p, size_t n) {
    const uint8_t *b = (const uint8_t *)p;
    buf.insert(buf.end(), b, b + n);
  }
  void u(uint64_t v, int n) {
    for (int i = 0; i < n; ++i) buf.push_back((uint8_t)(v >> (8 * i)));
  }
  void f32(float v) {
    uint32_t b;
    memcpy(&b, &v, 4);
    u(b, 4);
  }
  void f64(double v) {
    uint64_t b;
    memcpy(&b, &v, 8);
    u(b, 8);
  }
};

struct Reader {
  const uint8_t *p;
  size_t n, at = 0;
  bool ok = true;
  bool need(size_t k) {
    if (!ok || k > n - at) ok = false;
    return ok;
  }
  uint64_t u(int k) {
    if (!need((size_t)k)) return 0;
    uint64_t v = 0;
    for (int i = 0; i < k; ++i) v |= (uint64_t)p[at + i] << (8 * i);
    at += (size_t)k;
    return v;
  }
  double f64() {
    const uint64_t b = u(8);
    double v;
    memcpy(&v, &b, 8);
    return v;
  }
  const uint8_t *span(size_t k) {
    if (!need(k)) return nullptr;
    const uint8_t *q = p + at;
    at += k;
    return q;
  }
};

}  // namespace

struct seedq_container {
  std::vector<uint8_t> file;
  std::vector<seedq_rung> rungs;
  std::vector<double> theta;
  int32_t j_tie = -1;
  double q = 0.0;
  std::vector<std::string> names;
  // Host copies of the arrays (aligned, host byte order).
  std::vector<std::vector<float>> a, rho;
  std::vector<std::vector<int32_t>> cols;
  std::vector<std::vector<uint16_t>> vals;
  std::vector<seedq_container_tensor> t;
};

extern "C" {

seedq_status seedq_container_write(const char *path, const seedq_schedule *s, int32_t ntensors,
                                   const seedq_container_tensor *tensors) {
  if (!path || !s || !s->rungs || s->J < 1 || (s->J > 1 && !s->theta) || ntensors < 0 ||
      (ntensors > 0 && !tensors))
    return SEEDQ_ERR_INVALID_ARG;
  Writer w;
  w.bytes(kMagic, 8);
  w.u(1, 4);
  w.u((uint32_t)s->J, 4);
  for (int j = 0; j < s->J; ++j) {
    w.u((uint32_t)s->rungs[j].S, 4);
    w.u((uint32_t)s->rungs[j].k, 4);
  }
  for (int j = 0; j + 1 < s->J; ++j) w.f64(s->theta[j]);
  w.u((uint32_t)s->j_tie, 4);
  w.f64(s->q);
  for (int S = 8; S <= 16; ++S) w.u(seedq_lfsr_taps(S), 4);
  w.u((uint32_t)ntensors, 4);
  for (int i = 0; i < ntensors; ++i) {
    const seedq_container_tensor &t = tensors[i];
    if (t.rows < 1 || t.cols < 8 || !t.a || t.n_outliers < 0 || (t.n_outliers && (!t.outlier_cols ||
        !t.outlier_vals)) || (t.stream_bits && !t.stream))
      return SEEDQ_ERR_INVALID_ARG;
    const char *name = t.name ? t.name : "";
    const size_t nl = strlen(name);
    w.u(nl, 4);
    w.bytes(name, nl);
    w.u((uint64_t)t.rows, 8);
    w.u((uint64_t)t.cols, 8);
    for (int64_t c = 0; c < t.cols; ++c) w.f32(t.a[c]);
    w.u(t.rho ? 1 : 0, 4);
    if (t.rho)
      for (int64_t r = 0; r < t.rows; ++r) w.f32(t.rho[r]);
    w.u((uint64_t)t.tie_count, 8);
    w.u((uint32_t)t.n_outliers, 4);
    for (int o = 0; o < t.n_outliers; ++o) w.u((uint32_t)t.outlier_cols[o], 4);
    for (int64_t k = 0; k < t.rows * t.n_outliers; ++k) w.u(t.outlier_vals[k], 2);
    const uint64_t len = (t.stream_bits + 7) / 8;
    w.u(t.stream_bits, 8);
    w.u(len, 8);
    w.bytes(t.stream, len);
  }
  w.u(fnv1a(w.buf.data(), w.buf.size()), 8);
  FILE *f = fopen(path, "wb");
  if (!f) return SEEDQ_ERR_IO;
  const size_t put = fwrite(w.buf.data(), 1, w.buf.size(), f);
  const int closed = fclose(f);
  return (put == w.buf.size() && closed == 0) ? SEEDQ_OK : SEEDQ_ERR_IO;
}

seedq_status seedq_container_open(const char *path, seedq_container **out) {
  if (!path || !out) return SEEDQ_ERR_INVALID_ARG;
  *out = nullptr;
  FILE *f = fopen(path, "rb");
  if (!f) return SEEDQ_ERR_IO;
  seedq_container *c = new (std::nothrow) seedq_container;
  if (!c) {
    fclose(f);
    return SEEDQ_ERR_NOMEM;
  }
  uint8_t chunk[1 << 16];
  size_t got;
  while ((got = fread(chunk, 1, sizeof chunk, f)) > 0) c->file.insert(c->file.end(), chunk, chunk + got);
  const bool rerr = ferror(f) != 0;
  fclose(f);
  if (rerr) {
    delete c;
    return SEEDQ_ERR_IO;
  }
  seedq_status rc = SEEDQ_OK;
  const size_t n = c->file.size();
  if (n < 16 || memcmp(c->file.data(), kMagic, 8) != 0) rc = SEEDQ_ERR_FORMAT;
  Reader r{c->file.data(), n >= 8 ? n - 8 : 0};
  if (rc == SEEDQ_OK) {
    uint64_t h = 0;
    for (int i = 0; i < 8; ++i) h |= (uint64_t)c->file[n - 8 + i] << (8 * i);
    if (h != fnv1a(c->file.data(), n - 8)) rc = SEEDQ_ERR_FORMAT;
  }
  if (rc == SEEDQ_OK) {
    r.span(8);
    const uint64_t version = r.u(4), J = r.u(4);
    if (version != 1 || J < 1 || J > 9) rc = SEEDQ_ERR_FORMAT;
    for (uint64_t j = 0; rc == SEEDQ_OK && j < J; ++j) {
      seedq_rung g;
      g.S = (int32_t)r.u(4);
      g.k = (int32_t)r.u(4);
      c->rungs.push_back(g);
    }
    for (uint64_t j = 0; rc == SEEDQ_OK && j + 1 < J; ++j) c->theta.push_back(r.f64());
    c->j_tie = (int32_t)r.u(4);
    c->q = r.f64();
    for (int S = 8; S <= 16; ++S)
      if ((uint32_t)r.u(4) != seedq_lfsr_taps(S)) rc = SEEDQ_ERR_UNSUPPORTED;
  }
  uint64_t nt = rc == SEEDQ_OK ? r.u(4) : 0;
  if (!r.ok) rc = SEEDQ_ERR_FORMAT;
  for (uint64_t i = 0; rc == SEEDQ_OK && i < nt; ++i) {
    seedq_container_tensor t;
    memset(&t, 0, sizeof t);
    const uint64_t nl = r.u(4);
    const uint8_t *nm = r.span(nl);
    c->names.emplace_back(nm ? std::string((const char *)nm, nl) : std::string());
    t.rows = (int64_t)r.u(8);
    t.cols = (int64_t)r.u(8);
    if (!r.ok || t.rows < 1 || t.cols < 8 || t.rows > (1ll << 24) || t.cols > (1 << 16)) {
      rc = SEEDQ_ERR_FORMAT;
      break;
    }
    c->a.emplace_back((size_t)t.cols);
    for (int64_t k = 0; k < t.cols; ++k) {
      const uint32_t b = (uint32_t)r.u(4);
      memcpy(&c->a.back()[(size_t)k], &b, 4);
    }
    const uint64_t has_rho = r.u(4);
    c->rho.emplace_back(has_rho ? (size_t)t.rows : 0);
    for (int64_t k = 0; has_rho && k < t.rows; ++k) {
      const uint32_t b = (uint32_t)r.u(4);
      memcpy(&c->rho.back()[(size_t)k], &b, 4);
    }
    t.tie_count = (int64_t)r.u(8);
    const uint64_t no = r.u(4);
    if (!r.ok || no > 16) {
      rc = SEEDQ_ERR_FORMAT;
      break;
    }
    t.n_outliers = (int32_t)no;
    c->cols.emplace_back((size_t)no);
    for (uint64_t o = 0; o < no; ++o) c->cols.back()[(size_t)o] = (int32_t)r.u(4);
    c->vals.emplace_back((size_t)(no * (uint64_t)t.rows));
    for (uint64_t k = 0; k < no * (uint64_t)t.rows; ++k) c->vals.back()[(size_t)k] = (uint16_t)r.u(2);
    t.stream_bits = r.u(8);
    const uint64_t len = r.u(8);
    if (!r.ok || len != (t.stream_bits + 7) / 8) {
      rc = SEEDQ_ERR_FORMAT;
      break;
    }
    t.stream = r.span(len);
    if (!r.ok) rc = SEEDQ_ERR_FORMAT;
    c->t.push_back(t);
  }
  if (rc == SEEDQ_OK && (!r.ok || r.at != r.n)) rc = SEEDQ_ERR_FORMAT;
  if (rc != SEEDQ_OK) {
    delete c;
    return rc;
  }
  for (size_t i = 0; i < c->t.size(); ++i) {
    c->t[i].name = c->names[i].c_str();
    c->t[i].a = c->a[i].data();
    c->t[i].rho = c->rho[i].empty() ? nullptr : c->rho[i].data();
    c->t[i].outlier_cols = c->cols[i].empty() ? nullptr : c->cols[i].data();
    c->t[i].outlier_vals = c->vals[i].empty() ? nullptr : c->vals[i].data();
  }
  *out = c;
  return SEEDQ_OK;
}

seedq_status seedq_container_schedule(const seedq_container *c, seedq_schedule *s) {
  if (!c || !s) return SEEDQ_ERR_INVALID_ARG;
  s->J = (int32_t)c->rungs.size();
  s->rungs = c->rungs.data();
  s->theta = c->theta.empty() ? nullptr : c->theta.data();
  s->j_tie = c->j_tie;
  s->q = c->q;
  return SEEDQ_OK;
}

seedq_status seedq_container_count(const seedq_container *c, int32_t *n) {
  if (!c || !n) return SEEDQ_ERR_INVALID_ARG;
  *n = (int32_t)c->t.size();
  return SEEDQ_OK;
}

seedq_status seedq_container_get(const seedq_container *c, int32_t i, seedq_container_tensor *t) {
  if (!c || !t || i < 0 || (size_t)i >= c->t.size()) return SEEDQ_ERR_INVALID_ARG;
  *t = c->t[(size_t)i];
  return SEEDQ_OK;
}

seedq_status seedq_container_close(seedq_container *c) {
  delete c;
  return SEEDQ_OK;
}

}  // extern "C"
