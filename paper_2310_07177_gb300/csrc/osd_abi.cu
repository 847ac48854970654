// osd_abi.cu -- status strings and version of the C ABI declared in osd.h.
#include "osd.h"

extern "C" const char* osd_status_string(osd_status status) {
    switch (status) {
        case OSD_OK: return "OSD_OK";
        case OSD_ERR_INVALID_ARG: return "OSD_ERR_INVALID_ARG: null pointer, size, alignment or value out of range";
        case OSD_ERR_UNSUPPORTED: return "OSD_ERR_UNSUPPORTED: arguments beyond the library's limits";
        case OSD_ERR_CUDA: return "OSD_ERR_CUDA: a CUDA launch or API call failed";
        case OSD_ERR_TIMEOUT: return "OSD_ERR_TIMEOUT: a bounded device-side wait gave up";
    }
    return "OSD_ERR_UNKNOWN";
}

extern "C" int osd_abi_version(void) { return (2 << 16) | 5; }
