// lc_files.cu -- the file tier of the version store (§3.5): an append-only
// checkpoint directory with one CRC-checked record per persisted layer
// version, and the metadata-driven recovery that picks each layer's newest
// version at or before the failure step from the records alone and then
// reads only the blocks it picked.  Host code only; the device side of the
// recovery is lc_restore.  The on-disk format is documented in layercheck.h.
#include "layercheck.h"
#include "lc_host.h"

#include <errno.h>
#include <fcntl.h>
#include <sys/stat.h>
#include <sys/types.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <cstring>
#include <exception>
#include <set>
#include <string>
#include <thread>
#include <utility>
#include <vector>

namespace {

using lc::fail_status;

// ---------------------------------------------------------------------------
// CRC-32C.  The register is kept in reflected bit order: bit 31 holds the
// coefficient of x^0 and bit 0 that of x^31; kPoly is the Castagnoli
// polynomial without its x^32 term in that order.  Eight bytes are folded
// per step with eight 256-entry tables (the "slicing" table method): table
// k advances a byte through k further zero bytes.
// ---------------------------------------------------------------------------
constexpr uint32_t kPoly = 0x82F63B78u;

struct CrcTables {
    uint32_t t[8][256];
    CrcTables() {
        for (uint32_t b = 0; b < 256; ++b) {
            uint32_t r = b;
            for (int i = 0; i < 8; ++i) r = (r & 1u) ? (r >> 1) ^ kPoly : r >> 1;
            t[0][b] = r;
        }
        for (int k = 1; k < 8; ++k)
            for (uint32_t b = 0; b < 256; ++b) t[k][b] = (t[k - 1][b] >> 8) ^ t[0][t[k - 1][b] & 0xFFu];
    }
};

const CrcTables& crc_tables() {
    static const CrcTables tables;
    return tables;
}

inline uint32_t le32(const uint8_t* p) {
    return uint32_t(p[0]) | uint32_t(p[1]) << 8 | uint32_t(p[2]) << 16 | uint32_t(p[3]) << 24;
}

// The register after feeding n bytes (no initial or final inversion).
uint32_t crc_feed(uint32_t reg, const uint8_t* p, uint64_t n) {
    const CrcTables& T = crc_tables();
    while (n >= 8) {
        const uint32_t lo = reg ^ le32(p);
        const uint32_t hi = le32(p + 4);
        reg = T.t[7][lo & 0xFFu] ^ T.t[6][(lo >> 8) & 0xFFu] ^ T.t[5][(lo >> 16) & 0xFFu] ^ T.t[4][lo >> 24] ^
              T.t[3][hi & 0xFFu] ^ T.t[2][(hi >> 8) & 0xFFu] ^ T.t[1][(hi >> 16) & 0xFFu] ^ T.t[0][hi >> 24];
        p += 8;
        n -= 8;
    }
    while (n--) reg = (reg >> 8) ^ T.t[0][(reg ^ *p++) & 0xFFu];
    return reg;
}

// Product of two polynomials modulo the CRC polynomial (reflected order).
uint32_t poly_mulmod(uint32_t a, uint32_t b) {
    uint32_t prod = 0;
    for (int k = 0; k < 32; ++k) {          // coefficient of x^k in a is bit 31-k
        if (a & (0x80000000u >> k)) prod ^= b;
        b = (b & 1u) ? (b >> 1) ^ kPoly : b >> 1;   // b <- b * x
    }
    return prod;
}

// x^(8n) modulo the CRC polynomial, by square-and-multiply.
uint32_t x_pow_8n(uint64_t n) {
    uint32_t result = 0x80000000u;   // x^0
    uint32_t sq = 0x00800000u;       // x^8
    while (n) {
        if (n & 1u) result = poly_mulmod(result, sq);
        sq = poly_mulmod(sq, sq);
        n >>= 1;
    }
    return result;
}

// The CRC (initial and final inversion) of A followed by B from the CRCs of
// A and B: the inversions cancel, so crc(AB) = crc(A) * x^(8|B|) + crc(B).
uint32_t crc_concat(uint32_t crc_a, uint32_t crc_b, uint64_t len_b) {
    return poly_mulmod(x_pow_8n(len_b), crc_a) ^ crc_b;
}

uint32_t crc_serial(const uint8_t* p, uint64_t n, uint32_t crc) { return ~crc_feed(~crc, p, n); }

// Runs `worker` on this thread and on up to n - 1 more.  The workers take
// their items from one shared counter, so a thread that cannot be started
// is simply left out (the others take its share) and no joinable thread is
// abandoned while an exception unwinds.
template <typename F>
void run_on_threads(unsigned n, F&& worker) {
    std::vector<std::thread> pool;
    try {
        pool.reserve(n);
        for (unsigned t = 1; t < n; ++t) pool.emplace_back(worker);
    } catch (const std::exception&) {
    }
    worker();
    for (auto& t : pool) t.join();
}

// Pieces of kPiece bytes on up to hardware_concurrency threads, joined with
// crc_concat.
constexpr uint64_t kPiece = 64ull << 20;

uint32_t crc_parallel(const uint8_t* p, uint64_t n, uint32_t crc) {
    const uint64_t pieces = (n + kPiece - 1) / kPiece;
    const unsigned hw = std::max(1u, std::thread::hardware_concurrency());
    if (pieces < 2 || hw < 2) return crc_serial(p, n, crc);
    std::vector<uint32_t> part(pieces);
    std::atomic<uint64_t> next(0);
    auto worker = [&]() {
        for (uint64_t i; (i = next.fetch_add(1)) < pieces;) {
            const uint64_t a = i * kPiece, b = std::min(n, a + kPiece);
            part[i] = crc_serial(p + a, b - a, 0);
        }
    };
    run_on_threads(unsigned(std::min<uint64_t>(hw, pieces)), worker);
    for (uint64_t i = 0; i < pieces; ++i) {
        const uint64_t len = std::min(n, (i + 1) * kPiece) - i * kPiece;
        crc = crc_concat(crc, part[i], len);
    }
    return crc;
}

// ---------------------------------------------------------------------------
// format
// ---------------------------------------------------------------------------
constexpr size_t kRec = 64;
constexpr uint32_t kHeaderMagic = 0x484D434Cu;   // "LCMH"
constexpr uint32_t kRecordMagic = 0x5256434Cu;   // "LCVR"
constexpr uint32_t kFormat = 1;
constexpr uint64_t kBlockAlign = 4096;

inline void put32(uint8_t* p, uint32_t v) {
    for (int i = 0; i < 4; ++i) p[i] = uint8_t(v >> (8 * i));
}
inline void put64(uint8_t* p, uint64_t v) {
    for (int i = 0; i < 8; ++i) p[i] = uint8_t(v >> (8 * i));
}
inline uint64_t le64(const uint8_t* p) { return uint64_t(le32(p)) | uint64_t(le32(p + 4)) << 32; }

uint32_t layout_crc(int32_t nlayers, const uint64_t* layer_bytes) {
    std::vector<uint8_t> buf(size_t(nlayers) * 8);
    for (int32_t l = 0; l < nlayers; ++l) put64(buf.data() + 8 * l, layer_bytes[l]);
    return crc_serial(buf.data(), buf.size(), 0);
}

struct Header {
    int32_t nlayers;
    uint32_t layout;
};

void encode_header(const Header& h, uint8_t* out) {
    std::memset(out, 0, kRec);
    put32(out, kHeaderMagic);
    put32(out + 4, kFormat);
    put32(out + 8, uint32_t(h.nlayers));
    put32(out + 12, h.layout);
    put32(out + 60, crc_serial(out, 60, 0));
}

bool decode_header(const uint8_t* in, Header* h) {
    if (le32(in) != kHeaderMagic || le32(in + 4) != kFormat || le32(in + 60) != crc_serial(in, 60, 0)) return false;
    h->nlayers = int32_t(le32(in + 8));
    h->layout = le32(in + 12);
    return h->nlayers > 0;
}

void encode_record(const lc_manifest_record& r, uint8_t* out) {
    std::memset(out, 0, kRec);
    put32(out, kRecordMagic);
    put32(out + 4, uint32_t(r.layer));
    put64(out + 8, uint64_t(r.step));
    put64(out + 16, r.offset);
    put64(out + 24, r.bytes);
    put32(out + 32, r.block_crc);
    put32(out + 36, r.layout_crc);
    put32(out + 60, crc_serial(out, 60, 0));
}

bool decode_record(const uint8_t* in, lc_manifest_record* r) {
    if (le32(in) != kRecordMagic || le32(in + 60) != crc_serial(in, 60, 0)) return false;
    r->layer = int32_t(le32(in + 4));
    r->step = int64_t(le64(in + 8));
    r->offset = le64(in + 16);
    r->bytes = le64(in + 24);
    r->block_crc = le32(in + 32);
    r->layout_crc = le32(in + 36);
    r->intact = 1;
    return true;
}

// ---------------------------------------------------------------------------
// files
// ---------------------------------------------------------------------------
struct Fd {
    int fd = -1;
    Fd() = default;
    explicit Fd(int f) : fd(f) {}
    Fd(const Fd&) = delete;
    Fd& operator=(const Fd&) = delete;
    ~Fd() {
        if (fd >= 0) close(fd);
    }
};

std::string join(const char* dir, const char* name) {
    std::string s(dir);
    if (!s.empty() && s.back() != '/') s += '/';
    return s + name;
}

bool write_all(int fd, const uint8_t* p, uint64_t n, uint64_t off) {
    while (n) {
        const size_t want = size_t(std::min<uint64_t>(n, 1ull << 30));
        const ssize_t w = pwrite(fd, p, want, off_t(off));
        if (w < 0 && errno == EINTR) continue;
        if (w <= 0) return false;
        p += w;
        off += uint64_t(w);
        n -= uint64_t(w);
    }
    return true;
}

// Reads exactly n bytes; false on an error or a short file.
bool read_all(int fd, uint8_t* p, uint64_t n, uint64_t off) {
    while (n) {
        const size_t want = size_t(std::min<uint64_t>(n, 1ull << 30));
        const ssize_t r = pread(fd, p, want, off_t(off));
        if (r < 0 && errno == EINTR) continue;
        if (r <= 0) return false;
        p += r;
        off += uint64_t(r);
        n -= uint64_t(r);
    }
    return true;
}

// The manifest's header and its valid records (the log ends at the first
// short or invalid record).  `end` = byte offset just past the last valid
// record.
struct Manifest {
    Header h{};
    std::vector<lc_manifest_record> recs;
    uint64_t end = 0;
    bool torn = false;
};

lc_status read_manifest(int fd, const char* what, Manifest* m) {
    struct stat sb;
    if (fstat(fd, &sb) != 0) return fail_status(LC_ERR_INVALID_ARG, "%s: cannot stat the manifest", what);
    const uint64_t size = uint64_t(sb.st_size);
    std::vector<uint8_t> buf(size);
    if (size && !read_all(fd, buf.data(), size, 0))
        return fail_status(LC_ERR_INVALID_ARG, "%s: cannot read the manifest", what);
    if (size < kRec || !decode_header(buf.data(), &m->h))
        return fail_status(LC_ERR_STATE, "%s: the manifest header is missing or corrupt", what);
    uint64_t off = kRec;
    for (; off + kRec <= size; off += kRec) {
        lc_manifest_record r;
        if (!decode_record(buf.data() + off, &r)) break;
        m->recs.push_back(r);
    }
    m->end = off;
    m->torn = off != size;
    return LC_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
extern "C" uint32_t lc_crc32c(const void* data, uint64_t nbytes, uint32_t crc) {
    if (!data || nbytes == 0) return crc;
    return crc_parallel(static_cast<const uint8_t*>(data), nbytes, crc);
}

static lc_status lc_store_persist_dir_impl(lc_store* st, const char* dir, int32_t sync, uint64_t* bytes_written) {
    const char* what = "lc_store_persist_dir";
    lc::set_last_error("");
    if (bytes_written) *bytes_written = 0;
    if (!st || !dir || !*dir) return fail_status(LC_ERR_INVALID_ARG, "%s: NULL argument", what);
    if (mkdir(dir, 0755) != 0 && errno != EEXIST)
        return fail_status(LC_ERR_INVALID_ARG, "%s: cannot create %s: %s", what, dir, strerror(errno));
    const int32_t nl = lc::store_nlayers(st);
    const uint64_t* lb = lc::store_layer_bytes(st);
    const Header mine{nl, layout_crc(nl, lb)};
    Fd man(open(join(dir, "manifest.lcm").c_str(), O_RDWR | O_CREAT, 0644));
    if (man.fd < 0) return fail_status(LC_ERR_INVALID_ARG, "%s: cannot open the manifest: %s", what, strerror(errno));
    Manifest m;
    struct stat sb;
    if (fstat(man.fd, &sb) != 0) return fail_status(LC_ERR_INVALID_ARG, "%s: cannot stat the manifest", what);
    if (sb.st_size == 0) {
        uint8_t hb[kRec];
        encode_header(mine, hb);
        if (!write_all(man.fd, hb, kRec, 0) || (sync && fdatasync(man.fd) != 0))
            return fail_status(LC_ERR_INVALID_ARG, "%s: cannot write the manifest header", what);
        m.h = mine;
        m.end = kRec;
    } else {
        const lc_status rc = read_manifest(man.fd, what, &m);
        if (rc != LC_OK) return rc;
        if (m.h.nlayers != mine.nlayers || m.h.layout != mine.layout)
            return fail_status(LC_ERR_INVALID_ARG, "%s: %s holds another layout (%d layers)", what, dir,
                               m.h.nlayers);
        // a torn tail is dropped: the next record goes where it started
        if (m.torn && ftruncate(man.fd, off_t(m.end)) != 0)
            return fail_status(LC_ERR_INVALID_ARG, "%s: cannot cut the torn manifest tail", what);
    }
    std::set<std::pair<int32_t, int64_t>> have;
    for (const auto& r : m.recs) have.insert({r.layer, r.step});
    Fd blk(open(join(dir, "blocks.lcb").c_str(), O_RDWR | O_CREAT, 0644));
    if (blk.fd < 0) return fail_status(LC_ERR_INVALID_ARG, "%s: cannot open the block file: %s", what, strerror(errno));
    if (fstat(blk.fd, &sb) != 0) return fail_status(LC_ERR_INVALID_ARG, "%s: cannot stat the block file", what);
    // blocks past the last record (an append that never got its record) are overwritten
    uint64_t bend = 0;
    for (const auto& r : m.recs) bend = std::max(bend, r.offset + r.bytes);
    bend = (bend + kBlockAlign - 1) / kBlockAlign * kBlockAlign;
    uint64_t written = 0;
    const int64_t nv = lc_store_num_versions(st);
    for (int64_t i = 0; i < nv; ++i) {
        lc_version v;
        if (lc_store_get_version(st, i, &v) != LC_OK)
            return fail_status(LC_ERR_STATE, "%s: version %lld of the store is unreadable", what, (long long)i);
        if (!v.durable || have.count({v.layer, v.step})) continue;
        lc_manifest_record r;
        r.layer = v.layer;
        r.intact = 1;
        r.step = v.step;
        r.offset = bend;
        r.bytes = v.bytes;
        r.block_crc = lc_crc32c(v.host_ptr, v.bytes, 0);
        r.layout_crc = mine.layout;
        if (!write_all(blk.fd, static_cast<const uint8_t*>(v.host_ptr), v.bytes, bend) ||
            (sync && fdatasync(blk.fd) != 0))
            return fail_status(LC_ERR_INVALID_ARG, "%s: writing the block of layer %d step %lld failed: %s", what,
                               v.layer, (long long)v.step, strerror(errno));
        uint8_t rb[kRec];
        encode_record(r, rb);
        if (!write_all(man.fd, rb, kRec, m.end) || (sync && fdatasync(man.fd) != 0))
            return fail_status(LC_ERR_INVALID_ARG, "%s: writing a manifest record failed: %s", what, strerror(errno));
        m.end += kRec;
        bend = (bend + v.bytes + kBlockAlign - 1) / kBlockAlign * kBlockAlign;
        have.insert({v.layer, v.step});
        written += v.bytes;
    }
    if (bytes_written) *bytes_written = written;
    return LC_OK;
}

static lc_status lc_manifest_read_impl(const char* dir, int32_t verify_blocks, lc_manifest_record* out,
                                       int64_t cap, int64_t* n_out, int32_t* nlayers_out,
                                       uint32_t* layout_crc_out, int32_t* torn_out) {
    const char* what = "lc_manifest_read";
    lc::set_last_error("");
    if (!dir) return fail_status(LC_ERR_INVALID_ARG, "%s: dir is NULL", what);
    Fd man(open(join(dir, "manifest.lcm").c_str(), O_RDONLY));
    if (man.fd < 0) return fail_status(LC_ERR_INVALID_ARG, "%s: no manifest in %s", what, dir);
    Manifest m;
    const lc_status rc = read_manifest(man.fd, what, &m);
    if (rc != LC_OK) return rc;
    if (verify_blocks && !m.recs.empty()) {
        Fd blk(open(join(dir, "blocks.lcb").c_str(), O_RDONLY));
        struct stat bs;
        const uint64_t bsize = (blk.fd >= 0 && fstat(blk.fd, &bs) == 0) ? uint64_t(bs.st_size) : 0;
        std::vector<uint8_t> buf;
        for (auto& r : m.recs) {
            // a record may name bytes the file does not have (a truncated file)
            if (r.offset > bsize || r.bytes > bsize - r.offset) {
                r.intact = 0;
                continue;
            }
            buf.resize(size_t(r.bytes));
            r.intact = read_all(blk.fd, buf.data(), r.bytes, r.offset) &&
                       lc_crc32c(buf.data(), r.bytes, 0) == r.block_crc;
        }
    }
    if (out)
        for (int64_t i = 0; i < int64_t(m.recs.size()) && i < cap; ++i) out[i] = m.recs[size_t(i)];
    if (n_out) *n_out = int64_t(m.recs.size());
    if (nlayers_out) *nlayers_out = m.h.nlayers;
    if (layout_crc_out) *layout_crc_out = m.h.layout;
    if (torn_out) *torn_out = m.torn ? 1 : 0;
    return LC_OK;
}

static lc_status lc_store_load_dir_impl(lc_ctx* ctx, const char* dir, int64_t t_fail, lc_store** out,
                                        int64_t* layer_steps_out) {
    const char* what = "lc_store_load_dir";
    lc::set_last_error("");
    if (!ctx || !dir || !out) return fail_status(LC_ERR_INVALID_ARG, "%s: NULL argument", what);
    *out = nullptr;
    const int32_t nl = lc::ctx_nlayers(ctx);
    if (nl <= 0) return fail_status(LC_ERR_STATE, "%s: no layout registered", what);
    std::vector<uint64_t> lb(static_cast<size_t>(nl));
    for (int32_t l = 0; l < nl; ++l)
        if (lc_layer_block_bytes(ctx, l, &lb[size_t(l)]) != LC_OK) return LC_ERR_STATE;
    const uint32_t layout = layout_crc(nl, lb.data());
    Fd man(open(join(dir, "manifest.lcm").c_str(), O_RDONLY));
    if (man.fd < 0) return fail_status(LC_ERR_INVALID_ARG, "%s: no manifest in %s", what, dir);
    Manifest m;
    lc_status rc = read_manifest(man.fd, what, &m);
    if (rc != LC_OK) return rc;
    if (m.h.nlayers != nl || m.h.layout != layout)
        return fail_status(LC_ERR_INVALID_ARG, "%s: %s holds another layout (%d layers)", what, dir, m.h.nlayers);
    // the metadata pass: each layer's candidates, newest step first, later record first on a tie
    std::vector<std::vector<size_t>> cand(static_cast<size_t>(nl));
    for (size_t i = 0; i < m.recs.size(); ++i) {
        const lc_manifest_record& r = m.recs[i];
        if (r.layer < 0 || r.layer >= nl || r.step > t_fail || r.layout_crc != layout || r.bytes != lb[size_t(r.layer)])
            continue;
        cand[size_t(r.layer)].push_back(i);
    }
    for (auto& c : cand) {
        std::stable_sort(c.begin(), c.end(), [&](size_t a, size_t b) {
            if (m.recs[a].step != m.recs[b].step) return m.recs[a].step > m.recs[b].step;
            return a > b;
        });
    }
    for (int32_t l = 0; l < nl; ++l)
        if (cand[size_t(l)].empty())
            return fail_status(LC_ERR_NOT_FOUND, "%s: layer %d has no version at or before step %lld", what, l,
                               (long long)t_fail);
    Fd blk(open(join(dir, "blocks.lcb").c_str(), O_RDONLY));
    if (blk.fd < 0) return fail_status(LC_ERR_INVALID_ARG, "%s: no block file in %s", what, dir);
    uint64_t total = 0;
    for (uint64_t b : lb) total += b;
    lc_store* st = nullptr;
    rc = lc_store_create(&st, ctx, total, 0);
    if (rc != LC_OK) return rc;
    std::vector<uint8_t*> dst(static_cast<size_t>(nl));
    std::vector<int64_t> vidx(static_cast<size_t>(nl));
    for (int32_t l = 0; l < nl; ++l) dst[size_t(l)] = lc::store_append(st, l, &vidx[size_t(l)]);
    // the data pass: only the picked blocks are read, layers in parallel
    std::vector<int64_t> chosen(size_t(nl), -1);
    std::atomic<int32_t> next(0);
    auto worker = [&]() {
        for (int32_t l; (l = next.fetch_add(1)) < nl;) {
            for (size_t i : cand[size_t(l)]) {
                const lc_manifest_record& r = m.recs[i];
                if (read_all(blk.fd, dst[size_t(l)], r.bytes, r.offset) &&
                    crc_serial(dst[size_t(l)], r.bytes, 0) == r.block_crc) {
                    chosen[size_t(l)] = int64_t(i);
                    break;
                }
            }
        }
    };
    const unsigned hw = std::max(1u, std::thread::hardware_concurrency());
    run_on_threads(unsigned(std::min<int64_t>(hw, nl)), worker);
    for (int32_t l = 0; l < nl; ++l) {
        if (chosen[size_t(l)] < 0) {
            lc_store_destroy(st);
            return fail_status(LC_ERR_NOT_FOUND, "%s: layer %d has no intact version at or before step %lld", what,
                               l, (long long)t_fail);
        }
        const int64_t step = m.recs[size_t(chosen[size_t(l)])].step;
        lc::store_set_step(st, vidx[size_t(l)], step);
        if (layer_steps_out) layer_steps_out[l] = step;
    }
    *out = st;
    return LC_OK;
}

// The entry points: no C++ exception leaves the C ABI (a bad_alloc from a
// vector sized by the layout or the manifest becomes LC_ERR_OOM).
extern "C" lc_status lc_store_persist_dir(lc_store* st, const char* dir, int32_t sync, uint64_t* bytes_written) {
    try {
        return lc_store_persist_dir_impl(st, dir, sync, bytes_written);
    } catch (const std::exception& e) {
        return fail_status(LC_ERR_OOM, "lc_store_persist_dir: %s", e.what());
    }
}

extern "C" lc_status lc_manifest_read(const char* dir, int32_t verify_blocks, lc_manifest_record* out, int64_t cap,
                                      int64_t* n_out, int32_t* nlayers_out, uint32_t* layout_crc_out,
                                      int32_t* torn_out) {
    try {
        return lc_manifest_read_impl(dir, verify_blocks, out, cap, n_out, nlayers_out, layout_crc_out, torn_out);
    } catch (const std::exception& e) {
        return fail_status(LC_ERR_OOM, "lc_manifest_read: %s", e.what());
    }
}

extern "C" lc_status lc_store_load_dir(lc_ctx* ctx, const char* dir, int64_t t_fail, lc_store** out,
                                       int64_t* layer_steps_out) {
    try {
        return lc_store_load_dir_impl(ctx, dir, t_fail, out, layer_steps_out);
    } catch (const std::exception& e) {
        return fail_status(LC_ERR_OOM, "lc_store_load_dir: %s", e.what());
    }
}
